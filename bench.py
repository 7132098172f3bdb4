"""Benchmark of the gs-SGD compression step on GB300.

One step = the whole hot path for P simulated workers on one GPU: accumulate + Count
Sketch insert (fused), tree merge, median query + top-k, gather-and-zero.  The metric is
gradient coordinates per second, P * d * steps / time, for the ResNet-18-sized workload
(d = 11,173,962, P = 8, r = 5, c = 2^17, k = 11,200) unless --config names another.

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
import re
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
K1_SOURCE = os.path.join(ROOT, "paper_2108_06004_gb300", "csrc", "k_insert.cu")
PROFILE_DIR = os.path.join(ROOT, "profiles")
CPU_SAMPLE_D = 1 << 22   # coordinates per worker in one bounded oracle step (CPU baseline)
REF_BUDGET_S = 120.0     # oracle seconds for a whole --impl reference run
ORACLE_S_PER_COORD = 1.7e-7  # oracle seconds per worker-coordinate (sizes the reference samples)


VARIANTS = {
    "error_feedback": "S1-S6: per-worker momentum and error vectors, exact second round",
    "train": "S1-S7: as error_feedback, with the weight update fused into the second round",
    "heavymix": "S1-S6 with the HEAVYMIX selection in place of the top-k",
    "sketched_state": "momentum and error kept as r x c sketches; no per-worker state vectors",
}
HEAVYMIX_FILL_SEED = 0x5EED5EED
LR = 0.01


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="resnet18", choices=sorted(workloads.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--variant", default="error_feedback", choices=list(VARIANTS),
                    help="which form of the step to time (the default is the headline path)")
    ap.add_argument("--eager", action="store_true",
                    help="one library call per kernel instead of a captured plan per step")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-steps", action="store_true",
                    help="short run for a profiler: no e2e, no CPU baseline, no clocks")
    return ap.parse_args()


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


# ---- profile summary (ncu traffic) -------------------------------------------------------

def k1_traffic_per_launch(workload: str):
    """DRAM bytes per launch of the fused accumulate+insert kernel on this workload from the
    committed ncu summary (profiles/accumulate_insert_<workload>.md), if there is one and it
    was taken on the current kernel source (else None)."""
    try:
        text = open(os.path.join(PROFILE_DIR, f"accumulate_insert_{workload}.md")).read()
    except OSError:
        return None
    src = hashlib.sha256(open(K1_SOURCE, "rb").read()).hexdigest()[:16]
    m_sha = re.search(r"kernel source sha256\[:16\]:\s*`?([0-9a-f]{16})", text)
    m_tr = re.search(r"traffic per full launch \(bytes\):\s*`?([0-9.eE+]+)", text)
    if not m_sha or not m_tr or m_sha.group(1) != src:
        return None
    return float(m_tr.group(1))


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


# ---- our arm -----------------------------------------------------------------------------

def gpu_uuid(dev) -> str:
    import torch
    u = str(torch.cuda.get_device_properties(dev).uuid)
    return u if u.startswith("GPU-") else "GPU-" + u


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
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
    gs.load_library()

    w = workloads.get_config(args.config)
    P, d, r, c, k, rho = w.P, w.d, w.r, w.c, w.k, w.rho
    # Fresh gradients for each of the workload's steps (cycled if more steps are timed),
    # as many steps as fit a 24 GB pool.  Replicas on different ranks draw different
    # workers' gradients.  Large workloads are drawn on the device.
    step_bytes = P * d * 4
    nsteps_pool = max(1, min(w.steps, args.steps + args.warmup, (24 << 30) // step_bytes))
    host_gen = step_bytes <= (1 << 30)
    host_pool, dev_pool = [], []
    for t in range(nsteps_pool):
        if host_gen:
            gl = workloads.make_gradients(w, t, replica_workers(rank, P))
            host_pool.append([torch.from_numpy(g).pin_memory() for g in gl])
            dev_pool.append([g.to(dev, non_blocking=True) for g in host_pool[-1]])
        else:
            dev_pool.append([workloads.make_gradient_torch(w, t, q, torch.empty(d, device=dev))
                             for q in replica_workers(rank, P)])
    if not host_gen and not args.no_e2e and not args.profile_steps:
        host_pool = [[g.cpu().pin_memory() for g in dev_pool[0]]]
    us = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
    es = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
    sk = gs.gs_sketch_create(r, c, 20210813, P, 0)
    W = gs.gs_sketch_info(sk)["group_width"]
    groups = (P + W - 1) // W
    variant = args.variant
    ws_bytes = gs.gs_step_workspace_size(d, k)
    if variant == "heavymix":
        ws_bytes = max(ws_bytes, gs.gs_query_heavymix_workspace_size(d, k))
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    qws_bytes = gs.gs_query_topk_workspace_size(d, k)
    l2sq = torch.empty(1, dtype=torch.float64, device=dev)
    weights = torch.zeros(d, dtype=torch.float32, device=dev) if variant in ("train", "sketched_state") else None
    sk_u = sk_e = None
    if variant == "sketched_state":
        sk_u = gs.gs_sketch_create(r, c, 20210813, 1, 0)
        sk_e = gs.gs_sketch_create(r, c, 20210813, 1, 0)
        gs.gs_sketch_zero(sk_u)
        gs.gs_sketch_zero(sk_e)
    idx = torch.empty(k, dtype=torch.int64, device=dev)
    vals = torch.empty(k, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()

    # Plans (one CUDA graph per gradient buffer set, the insert phase timed by event nodes
    # inside the graph) unless --eager asks for one library call per kernel.  HEAVYMIX has
    # no plan form and always runs eagerly; the sketched state always runs as a plan.
    use_plan = (not args.eager or variant == "sketched_state") and variant != "heavymix"
    plans = []
    if use_plan:
        for grads in dev_pool:
            if variant == "sketched_state":
                plans.append(gs.gs_sketched_state_plan_create(sk, sk_u, sk_e, grads, d, rho, k, idx, vals, weights,
                                                              LR, ws, flags=gs.GS_PLAN_TIME_INSERT))
            else:
                plans.append(gs.gs_step_plan_create(sk, us, es, grads, d, rho, k, idx, vals, None, weights, LR, ws,
                                                    flags=gs.GS_PLAN_TIME_INSERT))
    k1_events = []

    def step(t, record):
        if use_plan:
            gs.gs_plan_launch(plans[t % nsteps_pool], stream)
            return
        grads = dev_pool[t % nsteps_pool]
        if variant == "sketched_state":
            gs.gs_sketched_state_step(sk, sk_u, sk_e, grads, d, rho, k, idx, vals, weights, LR, ws, None, stream)
            return
        gs.gs_sketch_zero(sk, stream)
        if record:
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
        gs.gs_accumulate_insert(sk, 0, us, es, grads, d, rho, stream)
        if record:
            e1.record(stream)
            k1_events.append((e0, e1))
        gs.gs_sketch_merge_tree(sk, P, stream)
        if variant == "heavymix":
            gs.gs_query_heavymix(sk, d, k, HEAVYMIX_FILL_SEED, idx, None, l2sq, ws, None, stream)
        else:
            gs.gs_query_topk(sk, d, k, idx, None, ws, qws_bytes, stream)
        if variant == "train":
            gs.gs_gather_zero_update(us, es, d, idx, k, vals, weights, LR, stream)
        else:
            gs.gs_gather_and_zero(us, es, d, idx, k, vals, stream)

    n_warm = max(args.warmup, len(plans))  # at least W steps, and every plan launched once
    for t in range(n_warm):
        step(t, False)
    torch.cuda.synchronize()

    clocks = None
    sampler = None
    if not args.profile_steps:
        sampler = ClockSampler(gpu_uuid(dev))
        sampler.start()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.mark_begin()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for t in range(args.steps):
        step(args.warmup + t, True)
    end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if sampler:
        sampler.mark_end()
    elapsed_ms = dist_max(start.elapsed_time(end), dev)
    if sampler:
        clocks = sampler.stop()

    # insert-phase durations of the timed steps: each covers all groups and row passes
    if use_plan:
        k1_ms = []
        for i, plan in enumerate(plans):
            n_timed = sum(1 for t in range(args.steps) if (args.warmup + t) % nsteps_pool == i)
            if n_timed:
                k1_ms += gs.gs_plan_insert_times(plan, n_timed)
    else:
        k1_ms = [a.elapsed_time(b) for a, b in k1_events]
    value = whole_job_rate(world, P, d, args.steps, elapsed_ms / 1e3)

    # Roofline of the dominant phase, the insert: 20 algorithmic HBM bytes per worker-
    # coordinate for the fused accumulate + insert (read g, u, e; write u, e); for the
    # sketched state, 4 (read g).  Tables larger than the L2 pass budget take several row
    # passes, each after the first re-reading e (or g): those bytes are reported as moved,
    # not counted as algorithmic.  One launch covers one group of W workers and one row pass,
    # so a phase is `groups` x `passes` launches.
    peaks, peak_kind = measured_peaks()
    rpp = gs.gs_sketch_info(sk)["rows_per_pass"]
    passes = -(-r // rpp)
    per_wc = 4.0 if variant == "sketched_state" else 20.0
    moved_wc = per_wc + 4.0 * (passes - 1)
    phase_s = (sum(k1_ms) / len(k1_ms)) / 1e3
    phase_bytes = per_wc * P * d
    k1_gbs = phase_bytes / phase_s / 1e9
    cells = d * r * groups
    roofline = {
        "kernel": ("k_accumulate_insert_coop (insert only" if variant == "sketched_state" else
                   "k_accumulate_insert_coop (fused S1+S2") + f", W={W}), the insert phase of a step: "
                  f"{groups} group(s) x {passes} row pass(es)",
        "row_passes": passes, "groups": groups, "algorithmic_bytes_per_worker_coord": per_wc,
        "moved_bytes_per_worker_coord": moved_wc,
        "bound": "hbm", "achieved": round(k1_gbs, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
        "frac": round(k1_gbs / peaks["hbm_gbs"], 4), "peak_source": peak_kind,
        "frac_of_nominal_8000_GBps": round(k1_gbs / 8000.0, 4),
        "traffic": k1_traffic_per_launch(w.name) if variant != "sketched_state" and groups * passes == 1 else None,
        "algorithmic_bytes_per_launch": phase_bytes / (groups * passes) if passes == 1 else None,
        "algorithmic_bytes_per_phase": phase_bytes,
        "avg_launch_ms": round(sum(k1_ms) / len(k1_ms) / (groups * passes), 4),
        "avg_phase_ms": round(sum(k1_ms) / len(k1_ms), 4),
        "timed_phases": len(k1_ms),
        "timing": "event-record nodes inside the step's CUDA graph" if use_plan else "CUDA events around the call",
        "co_bound": {"kind": "SM->L2 payload: cell reductions (4*r B per worker-coordinate) + u, e stores "
                             "(8 B per worker-coordinate; none for the sketched state)",
                     "cell_updates_per_phase": cells,
                     "achieved_G_cells_per_s": round(cells / phase_s / 1e9, 1),
                     "probe_peak_G_cells_per_s": 134.5,
                     "sm_to_l2_payload_GBps": round(P * d * (4 * r + (0 if variant == "sketched_state" else 8))
                                                    / phase_s / 1e9, 1)},
        "step_share": round(sum(k1_ms) / elapsed_ms, 3),
    }

    # end to end through the public API with host buffers: a host plan per gradient set (the
    # uploads where needed, the step and the download of idx and vals are one graph), then a
    # stream synchronisation so that the host can read the step's result
    e2e = None
    if not args.no_e2e and not args.profile_steps and variant == "error_feedback":
        grad_dev = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(P)]
        idx_h = torch.empty(k, dtype=torch.int64).pin_memory()
        vals_h = torch.empty(k, dtype=torch.float32).pin_memory()
        hplans = []
        if use_plan:
            hplans = [gs.gs_step_host_plan_create(sk, us, es, hb, grad_dev, d, rho, k, idx_h, vals_h, ws)
                      for hb in host_pool]

        def host_step(t):
            if use_plan:
                gs.gs_plan_launch(hplans[t % len(hplans)], stream)
                stream.synchronize()
            else:
                gs.gs_step_host(sk, us, es, host_pool[t % len(host_pool)], grad_dev, d, rho, k, idx_h, vals_h, ws,
                                None, stream)

        for t in range(max(args.warmup, len(hplans))):  # every plan once, at least W steps
            host_step(t)
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for t in range(args.steps):
            host_step(args.warmup + t)
        torch.cuda.synchronize()
        e2e_s = time.perf_counter() - t0
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        e2e_s = dist_max(e2e_s, dev)
        for hp in hplans:
            gs.gs_plan_destroy(hp)
        e2e = {"value": whole_job_rate(world, P, d, args.steps, e2e_s), "unit": UNIT, "h2d_bytes_per_step": P * d * 4,
               "d2h_bytes_per_step": k * (8 + 4), "ms_per_step": round(e2e_s * 1e3 / args.steps, 4),
               "call": "gs_step_host_plan_create + gs_plan_launch" if use_plan else "gs_step_host"}

    for plan in plans:
        gs.gs_plan_destroy(plan)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.profile_steps \
            and variant == "error_feedback":
        cpu = cpu_baseline(w, steps=2)

    gs.gs_sketch_destroy(sk)
    for extra in (sk_u, sk_e):
        if extra:
            gs.gs_sketch_destroy(extra)
    # insert (one per group and row pass), merge, query + selection (7; HEAVYMIX 10), then
    # the gather (sketched state: cell accumulate, take, query_at, two sparse inserts, update)
    # the top-k query adds its repair check where it prunes rows (d >= 2^22, r >= 3, c a power of two)
    prunes = variant != "heavymix" and d >= (1 << 22) and r >= 3 and (c & (c - 1)) == 0
    launches_per_step = groups * passes + 1 + (10 if variant == "heavymix" else 7) + (1 if prunes else 0) + \
        (6 if variant == "sketched_state" else 1)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(elapsed_ms / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": w.name, "variant": variant, "launch": "plan" if use_plan else "eager",
                   "warmup_steps_run": n_warm, "d": d, "P": P, "r": r, "c": c, "k": k, "rho": rho, "group_width": W,
                   "parallelism": f"replicas{world}" if world > 1 else "single-gpu",
                   "l2": f"inputs larger than L2 ({P * d * 12 / 1e9:.2f} GB of g,u,e streamed per step)",
                   "d_steps_per_s": world * d * args.steps / (elapsed_ms / 1e3)},
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
    }
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
