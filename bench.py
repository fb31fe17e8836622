#!/usr/bin/env python3
"""Benchmark of the AGS optimizer step (one step = the reduction pass + the
update pass over a whole parameter set) on GB300.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload resnet50]
  python bench.py --impl reference ...   # the CPU oracle on the host cores

Prints ONE JSON line.  `value` is parameters updated per second over the whole
job, device-resident inputs; `e2e` is the same metric through the C ABI with
the replica gradients copied in from pinned host memory and the step record and
per-layer statistics copied back inside the timed region.  `secondary` holds the
same step timed on the VGG-16 parameter set (the other set the roofline target
names), and `cpu_baseline` the CPU oracle on all host cores, with its
single-threaded figure beside it.  Under torchrun every rank runs its own
replica step on its own GPU (no collective on the data path: one optimizer step
has nothing to exchange once the K replicas are local), and the time is the max
over ranks.
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
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "AGS optimizer steps/sec and params/sec; achieved HBM GB/s vs ~8 TB/s peak"
UNIT = "params/s"
FALLBACK_HBM_GBS = 6800.0


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="resnet50")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--soak-s", type=float, default=1.0,
                    help="untimed load before the timed steps, so clock samples see load")
    ap.add_argument("--cpu-sample-s", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-secondary", dest="secondary", action="store_false",
                    help="skip the second parameter set (VGG-16) timed after the headline one")
    ap.add_argument("--granularity", default="tensor", choices=["tensor", "element"],
                    help="gradscale per tensor (default) or per element (Algorithm 1's line "
                         "read literally; the update then reads a scale per parameter)")
    ap.add_argument("--no-momentum", dest="momentum", action="store_false",
                    help="steps without a momentum buffer (w -= lr * d)")
    ap.add_argument("--step-kind", default="ags", choices=list(STEP_KINDS),
                    help="ags: Algorithm 1 steps (the gradscale refreshed once, in warm-up); "
                         "refresh: every step also refreshes the gradscale (UpdateGradScale fused "
                         "into pass 1, precise norms); lars: the LARS rule (precise norms, w read "
                         "in pass 1)")
    return ap.parse_args()


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(ms: float, device="cuda") -> float:
    """The job's time: the slowest rank's (every rank calls this; one process: unchanged)."""
    import torch
    import torch.distributed as dist
    if not dist.is_initialized() or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(params_per_rank: int, steps: int, world_size: int, t_max_ms: float) -> float:
    """Parameters updated per second by the whole job: every rank runs its own replica of the
    step (weak scaling), and the job takes as long as its slowest rank."""
    return world_size * params_per_rank * steps / (t_max_ms / 1e3)


# ---------------------------------------------------------------------------
# bytes per parameter (fp32)
# ---------------------------------------------------------------------------

LARS_TRUST = 1e-3  # trust coefficient of the LARS steps timed here
# step kind -> (reads w in pass 1, refreshes the gradscale every step)
STEP_KINDS = {"ags": (False, False), "refresh": (False, True), "lars": (True, False),
              "update-scale": (False, False), "sharded": (False, False)}


def pass1_bytes_per_param(K: int, read_w: bool = False) -> int:
    """Reduction pass: read K replicas (and w for LARS), write the mean over replica 0 (K > 1)."""
    return 4 * K + (4 if K > 1 else 0) + (4 if read_w else 0)


def pass2_bytes_per_param(with_momentum=True, per_element=False) -> int:
    """Update pass: read gbar, w, m; write w, m (no momentum buffer: read gbar, w; write w).  A
    per-element gradscale is read too (in a scaled step)."""
    return (20 if with_momentum else 12) + (4 if per_element else 0)


def step_design_bytes_per_param(K: int, read_w: bool = False, with_momentum=True,
                                per_element=False) -> int:
    """What the two passes move as built: pass 1 plus pass 2 (the mean is written over
    replica 0 and read back by the update, as an in-place all-reduce would leave it)."""
    return pass1_bytes_per_param(K, read_w) + pass2_bytes_per_param(with_momentum, per_element)


def step_min_bytes_per_param(K: int, read_w: bool = False, with_momentum=True,
                             per_element=False) -> int:
    """Algorithmic minimum of one step: read K replicas, w, m; write w, m (LARS: w is read
    once more, since its norm sets the coefficient before the update; no momentum buffer: 8
    bytes less; a per-element gradscale: 4 more)."""
    return (4 * K + 16 + (4 if read_w else 0) - (0 if with_momentum else 8)
            + (4 if per_element else 0))


def scale_elem_bytes_per_param() -> int:
    """UpdateGradScale element-wise: read g_small and g_large, write the scale."""
    return 12


# ---------------------------------------------------------------------------
# clocks (nvidia-smi sampled while the GPU is loaded)
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for _, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for name, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# ncu-measured DRAM traffic of the dominant kernel (committed summary)
# ---------------------------------------------------------------------------

def _kernel_source_sha() -> str:
    path = os.path.join(ROOT, "paper_2603_18112_gb300", "csrc", "tula_ags.cu")
    return hashlib.sha256(open(path, "rb").read()).hexdigest()[:16]


def _ncu_traffic(kernel: str, workload: str, params: int):
    """Bytes per launch from profiles/dram_traffic.txt if it was taken on the current
    kernel source; scaled by parameters when the capture was a smaller case."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    sha = _kernel_source_sha()
    for line in open(path):
        f = line.split()
        if len(f) >= 5 and not line.startswith("#") and f[0] == kernel and f[1] == workload \
                and f[2] == sha:
            captured_params = int(f[3])
            return float(f[4]) * params / captured_params
    return None


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline leg and --impl reference)
# ---------------------------------------------------------------------------

def _host_inputs(wl, frac=1.0):
    import numpy as np
    import torch

    from paper_2603_18112_gb300 import workloads as W
    pset = wl.pset
    if frac < 1.0:
        keep, tot = [], 0
        budget = frac * pset.n_params
        for s, k in zip(pset.shapes, pset.kinds):
            if tot >= budget and keep:
                break
            keep.append((s, k))
            tot += int(np.prod(s))
        sub = W.ParamSet(pset.name + "-sample")
        for s, k in keep:
            sub.add(s, k)
        pset = sub
    buf = W.allocate(wl, "cpu", pset=pset)
    torch.set_num_threads(max(1, os.cpu_count() or 1))
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    w = W.to_numpy(buf.w)
    m = W.to_numpy(buf.m)
    g = [W.to_numpy(buf.g[k]) for k in range(wl.K)]
    return pset, w, m, g


def host_cores() -> int:
    """Threads the all-cores oracle runs on: the host's CPU count (bounded by what the oracle's
    OpenMP build can use)."""
    import oracle as O
    return max(1, min(os.cpu_count() or 1, O.max_threads()))


def _oracle_steps(wl, w, m, g, steps, kind="ags", threads=None):
    import numpy as np

    import oracle as O
    hp = O.OracleHP(K=wl.K, s_max=wl.smax, rule=O.RULE_LARS if kind == "lars" else O.RULE_AGS,
                    lars_trust=LARS_TRUST)
    hp.refresh_scale = kind == "refresh"
    scale = np.ones(len(w), np.float32)
    state = O.new_state()
    t0 = time.perf_counter()
    for _ in range(steps):
        O.ags_step(w, m, g, wl.lr, wl.momentum, wl.weight_decay, hp, scale=scale, state=state,
                   threads=threads)
    return time.perf_counter() - t0


def _timed_oracle(wl, pset, w, m, g, budget_s, kind, threads):
    t1 = _oracle_steps(wl, w, m, g, 1, kind, threads)
    steps = max(1, min(50, int(budget_s / max(t1, 1e-6))))
    t = _oracle_steps(wl, w, m, g, steps, kind, threads)
    return pset.n_params * steps / t, steps


def cpu_baseline(wl, budget_s, kind="ags"):
    """The oracle as it stands on the host: a bounded number of full optimizer steps over the
    same parameter set, on all host cores (its per-tensor parts in parallel, the combine in
    tensor order; bitwise the single-threaded result) and on one core."""
    pset, w, m, g = _host_inputs(wl)
    cores = host_cores()
    v_all, s_all = _timed_oracle(wl, pset, w, m, g, budget_s / 2, kind, cores)
    v_one, s_one = _timed_oracle(wl, pset, w, m, g, budget_s / 2, kind, None)
    what = (f"full steps of the {wl.name} parameter set ({pset.n_params} params, "
            f"{pset.n_tensors} tensors, K={wl.K}) on the host, C oracle")
    return {"value": v_all, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{s_all} {what}, per-tensor parts on {cores} threads",
            "host_cpu_count": os.cpu_count(),
            "single_thread": {"value": v_one, "unit": UNIT, "cores": 1,
                              "sample": f"{s_one} {what}, one thread"}}


def run_reference(args, wl):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    pset_full = wl.pset
    kind = args.step_kind
    if kind == "update-scale":
        raise SystemExit("--impl reference times optimizer steps, not --step-kind update-scale")
    if STEP_KINDS[kind][1] and wl.K == 1:
        raise SystemExit("--step-kind refresh needs K > 1 (g_small is replica 0)")
    _, w, m, g = _host_inputs(wl)
    cores = host_cores()
    t1 = _oracle_steps(wl, w, m, g, 1, kind, cores)
    total = args.steps + args.warmup
    frac = min(1.0, 120.0 / max(1e-9, total * t1))
    if frac < 1.0:
        pset, w, m, g = _host_inputs(wl, frac)
    else:
        pset = pset_full
    _oracle_steps(wl, w, m, g, args.warmup, kind, cores)
    t = _oracle_steps(wl, w, m, g, args.steps, kind, cores)
    value = pset.n_params * args.steps / t
    sample = (f"each step: the C oracle, per-tensor parts on {cores} threads, over "
              f"{'all' if frac >= 1.0 else 'the first'} {pset.n_tensors} tensors "
              f"({pset.n_params} of {pset_full.n_params} params) of the {wl.name} set, K={wl.K}")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * t / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": _config(wl, pset_full, kind),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": sample, "host_cpu_count": os.cpu_count()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


STEP_KIND_TEXT = {
    "ags": "Algorithm 1 step (AGS rule, per-tensor gradscale)",
    "update-scale": "UpdateGradScale of Algorithm 1 alone, element-wise (g_small = replica 1, "
                    "g_large = replica 0): not a step",
    "refresh": "Algorithm 1 step that also refreshes the gradscale (UpdateGradScale, g_small = "
               "replica 0)",
    "lars": "LARS rule step (coefficient 0.001 |w| / |gbar|)",
    "sharded": "Algorithm 1 step sharded over 2 ranks run one after the other on one GPU (pass 1 "
               "of each shard, the shares of |G|^2 summed by an integer add on the GPU, then the "
               "rest of each shard): the same results as the whole step",
}


def _config(wl, pset, kind="ags", per_elem=False, momentum=True):
    step = STEP_KIND_TEXT[kind]
    if per_elem:
        step += "; gradscale per element"
    if not momentum:
        step += "; no momentum buffer"
    return {"workload": f"{wl.name} parameter set, K={wl.K} replica gradient buffers",
            "step": step,
            "params": pset.n_params, "tensors": pset.n_tensors, "K": wl.K,
            "global_batch": None, "seq_len": None, "parallelism": "replicas only (1 step per GPU)",
            "l2": "inputs larger than L2 (no flush): "
                  f"{step_min_bytes_per_param(wl.K, STEP_KINDS[kind][0]) * pset.n_params / 1e9:.2f}"
                  " GB touched per step vs 126 MB L2"}


# ---------------------------------------------------------------------------
# GPU timing
# ---------------------------------------------------------------------------

SECONDARY = "vgg16"  # the other parameter set the >= 80 % roofline target names


def secondary_record(name, args, kind, stream, peak):
    """The step on a second parameter set, timed the same way as the headline (steps back to
    back on one stream, CUDA events; then the same steps again with events at the kernel
    boundaries for the per-kernel fractions).  Inputs are device-resident; its tensors are
    freed before returning."""
    import torch

    from paper_2603_18112_gb300 import tula_ags as T
    from paper_2603_18112_gb300 import workloads as W
    wl = W.workload(name)
    read_w, refresh = STEP_KINDS[kind]
    if refresh and wl.K == 1:
        return None
    N, K = wl.pset.n_params, wl.K
    buf = W.allocate(wl, "cuda")
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    torch.cuda.synchronize()
    step = T.AGSOptimizerStep(buf.w, buf.g, buf.m, s_max=wl.smax,
                              rule=T.TULA_RULE_LARS if kind == "lars" else T.TULA_RULE_AGS,
                              lars_trust=LARS_TRUST)
    steps = max(1, min(args.steps, 100))
    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            step.step(wl.lr, wl.momentum, wl.weight_decay,
                      refresh_scale=refresh or (kind == "ags" and i == 0 and K > 1), stream=stream)
    stream.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(steps):
            step.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=refresh, stream=stream)
        t1.record(stream)
    stream.synchronize()
    ms = t0.elapsed_time(t1) / steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(steps)]
    with torch.cuda.stream(stream):
        for e5 in evs:  # recorded once by torch, so that it times them
            for e in e5:
                e.record(stream)
        for e5 in evs:
            step.set_trace_events(e5)
            step.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=refresh, stream=stream)
    step.set_trace_events(None)
    torch.cuda.synchronize()
    red = statistics.fmean(e[0].elapsed_time(e[1]) for e in evs)
    upd = statistics.fmean(e[2].elapsed_time(e[3]) for e in evs)
    p1 = pass1_bytes_per_param(K, read_w) * N
    p2 = pass2_bytes_per_param() * N
    step_gbs = step_min_bytes_per_param(K, read_w) * N / (ms / 1e3) / 1e9
    out = {"workload": f"{name} parameter set, K={K} replica gradient buffers",
           "params": N, "tensors": wl.pset.n_tensors, "steps": steps, "ms_per_step": ms,
           "value": N / (ms / 1e3), "unit": UNIT,
           "k_reduce": {"ms_per_launch": red, "bytes_per_launch": p1,
                        "frac": p1 / (red / 1e3) / 1e9 / peak},
           "k_update": {"ms_per_launch": upd, "bytes_per_launch": p2,
                        "frac": p2 / (upd / 1e3) / 1e9 / peak},
           "step_hbm": {"algorithmic_bytes_per_param": step_min_bytes_per_param(K, read_w),
                        "achieved_gbs": step_gbs, "frac": step_gbs / peak,
                        "frac_of_8tbs": step_gbs / 8000.0},
           "l2": "inputs larger than L2 (no flush)"}
    del step, buf
    torch.cuda.empty_cache()
    return out


def run_ours(args, wl):
    import torch
    import torch.distributed as dist

    from paper_2603_18112_gb300 import build as B
    from paper_2603_18112_gb300 import tula_ags as T
    from paper_2603_18112_gb300 import workloads as W

    ws, rank, local = _dist()
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    if not B.LIB.exists():
        B.build()
    T.lib()

    pset = wl.pset
    N = pset.n_params
    K = wl.K
    kind = args.step_kind
    read_w, refresh = STEP_KINDS[kind]
    if refresh and K == 1:
        raise SystemExit("--step-kind refresh needs K > 1 (g_small is replica 0)")
    per_elem = args.granularity == "element"
    mu = wl.momentum if args.momentum else 0.0
    buf = W.allocate(wl, "cuda", with_momentum=args.momentum)
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    stream = torch.cuda.Stream()
    scale_elem = None
    if per_elem:  # a per-element gradscale in [0.5, 2]
        gen = torch.Generator(device="cuda")
        gen.manual_seed(wl.seed * 7919 + 5)
        scale_elem = [torch.rand(t.shape, generator=gen, device="cuda") * 1.5 + 0.5 for t in buf.w]
    torch.cuda.synchronize()
    # LARS with a trust coefficient of 1 moves w by about |w| each step: on one gradient reused
    # for thousands of steps the weights overflow within ~120 steps, and every tile then takes
    # the exact-fp64 fallback of the precise norms.  0.001 keeps them bounded.
    step = T.AGSOptimizerStep(buf.w, buf.g, buf.m if args.momentum else None, s_max=wl.smax,
                              rule=T.TULA_RULE_LARS if kind == "lars" else T.TULA_RULE_AGS,
                              lars_trust=LARS_TRUST,
                              granularity=(T.TULA_SCALE_PER_ELEMENT if per_elem
                                           else T.TULA_SCALE_PER_TENSOR),
                              scale_elem=scale_elem)

    def one_step():
        step.step(wl.lr, mu, wl.weight_decay, refresh_scale=refresh, stream=stream)

    def barrier():
        if ws > 1:
            dist.barrier()

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            # the first warm-up step refreshes the gradscale (UpdateGradScale needs K > 1)
            step.step(wl.lr, mu, wl.weight_decay,
                      refresh_scale=refresh or (kind == "ags" and i == 0 and K > 1 and not per_elem),
                      stream=stream)
    stream.synchronize()

    # per-step pass boundaries, recorded by the library on `stream`
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    with torch.cuda.stream(stream):
        for trio in evs:
            for e in trio:
                e.record(stream)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)

    sampler = ClockSampler(local)
    sampler.start()
    # untimed load so the clock samples are taken under load (part of the warm-up)
    soak = 0
    t0 = time.time()
    with torch.cuda.stream(stream):
        while time.time() - t0 < args.soak_s:
            for _ in range(20):
                one_step()
            soak += 20
            stream.synchronize()
    barrier()
    torch.cuda.synchronize()
    # The timed steps: back to back, nothing between the kernels of consecutive steps.
    launches0 = T.tula_ags_launch_count()
    with torch.cuda.stream(stream):
        t_start.record(stream)
        for _ in range(args.steps):
            one_step()
        t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = T.tula_ags_launch_count() - launches0
    # Host time per call: 50 steps issued after a synchronize, timed on the host up to the
    # return of the last call (the launch queue holds them all, so the host never waits on
    # the GPU unless it is the faster side).  Once through the plan the timed steps use, once
    # through tula_ags_step, which checks every pointer and builds the launch tables per call.
    def host_us_per_call(fn):
        torch.cuda.synchronize()
        h0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for _ in range(50):
                fn()
        us = (time.perf_counter() - h0) / 50 * 1e6
        torch.cuda.synchronize()
        return us

    host_us = host_us_per_call(one_step)
    direct = T.AGSOptimizerStep(buf.w, buf.g, buf.m if args.momentum else None, s_max=wl.smax,
                                rule=step.hp.rule, lars_trust=LARS_TRUST,
                                granularity=step.hp.granularity, scale_elem=scale_elem,
                                plan=False)
    host_us_direct = host_us_per_call(
        lambda: direct.step(wl.lr, mu, wl.weight_decay, refresh_scale=refresh, stream=stream))
    del direct
    peak, peak_kind = _peaks()
    secondary = (secondary_record(SECONDARY, args, kind, stream, peak)
                 if args.secondary and wl.name != SECONDARY and not per_elem and args.momentum
                 else None)
    clocks = sampler.stop()
    elapsed_ms = t_start.elapsed_time(t_end)
    # Per-pass times: the same steps again, with the library recording events at the pass
    # boundaries on the launching stream (an event between kernels stops the next kernel from
    # starting early, so these are slightly pessimistic).
    with torch.cuda.stream(stream):
        for trio in evs:
            step.set_trace_events(trio)
            one_step()
    step.set_trace_events(None)
    torch.cuda.synchronize()
    # kernel boundaries: [0] k_reduce [1] k_combine (pass 1) [2] k_update [3] k_combine [4]
    t_red = [e[0].elapsed_time(e[1]) for e in evs]
    t_cmb1 = [e[1].elapsed_time(e[2]) for e in evs]
    t_upd = [e[2].elapsed_time(e[3]) for e in evs]
    t_cmb2 = [e[3].elapsed_time(e[4]) for e in evs]

    t_max_ms = max_over_ranks(elapsed_ms)

    # ---- end to end through the C ABI with host buffers -------------------
    e2e = None
    h2d = K * buf.total * 4
    d2h = (T.TULA_STATE_LEN + T.TULA_STATS_LEN * pset.n_tensors) * 8
    host_g = [torch.empty(buf.total, dtype=torch.float32, pin_memory=True) for _ in range(K)]
    for k in range(K):
        host_g[k].copy_(buf.g_flats[k][:buf.total])
    host_state = torch.empty(T.TULA_STATE_LEN, dtype=torch.float64, pin_memory=True)
    host_stats = torch.empty(pset.n_tensors, T.TULA_STATS_LEN, dtype=torch.float64,
                             pin_memory=True)
    torch.cuda.synchronize()
    barrier()
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e_start.record(stream)
        for _ in range(args.e2e_steps):
            for k in range(K):
                buf.g_flats[k][:buf.total].copy_(host_g[k], non_blocking=True)
            one_step()
            host_state.copy_(step.state, non_blocking=True)
            host_stats.copy_(step.stats, non_blocking=True)
        e_end.record(stream)
    stream.synchronize()
    e2e_ms = max_over_ranks(e_start.elapsed_time(e_end))
    e2e = {"value": job_throughput(N, args.e2e_steps, ws, e2e_ms), "unit": UNIT,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": args.e2e_steps}

    if rank != 0:
        dist.destroy_process_group()
        return

    p1_avg_ms = statistics.fmean(t_red)
    p2_avg_ms = statistics.fmean(t_upd)
    p1_bytes = pass1_bytes_per_param(K, read_w) * N
    p2_bytes = pass2_bytes_per_param(args.momentum, per_elem) * N
    achieved = p1_bytes / (p1_avg_ms / 1e3) / 1e9
    ms_per_step = t_max_ms / args.steps
    smin = step_min_bytes_per_param(K, read_w, args.momentum, per_elem)
    sdes = step_design_bytes_per_param(K, read_w, args.momentum, per_elem)
    step_gbs = smin * N / (ms_per_step / 1e3) / 1e9
    red_name = "k_reduce" if kind == "ags" else f"k_reduce_{kind}"
    traffic = _ncu_traffic(red_name, wl.name, N)
    line = {
        "metric": METRIC, "value": job_throughput(N, args.steps, ws, t_max_ms), "unit": UNIT,
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "steps_per_s": 1e3 / ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": _config(wl, pset, kind, per_elem, args.momentum),
        "roofline": {"bound": "hbm",
                     "kernel": "k_reduce (replica mean + tile norms"
                               + (")" if kind == "ags" else ", precise norms)"),
                     "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "traffic": traffic, "bytes_per_launch": p1_bytes,
                     "ms_per_launch": p1_avg_ms},
        "update_pass": {"kernel": "k_update (scaled momentum-SGD)", "bytes_per_launch": p2_bytes,
                        "traffic": _ncu_traffic("k_update" + ("_per_element" if per_elem else "")
                                                + ("" if args.momentum else "_no_momentum"),
                                                wl.name, N),
                        "ms_per_launch": p2_avg_ms,
                        "achieved_gbs": p2_bytes / (p2_avg_ms / 1e3) / 1e9,
                        "frac": p2_bytes / (p2_avg_ms / 1e3) / 1e9 / peak},
        "combine_ms": {"after_reduce": statistics.fmean(t_cmb1),
                       "after_update": statistics.fmean(t_cmb2)},
        "step_hbm": {"algorithmic_bytes_per_param": smin,
                     "achieved_gbs": step_gbs, "frac": step_gbs / peak,
                     "frac_of_8tbs": step_gbs / 8000.0,
                     "design_bytes_per_param": sdes,
                     "design_gbs": sdes * N / (ms_per_step / 1e3) / 1e9},
        "e2e": e2e,
        "host_us_per_call": host_us,
        "host_us_per_call_direct": host_us_direct,
        "secondary": [secondary] if secondary else [],
        "gpu_launches": launches,
        "clocks": clocks,
        "soak_steps": soak,
    }
    if not args.no_cpu_baseline and ws == 1:
        line["cpu_baseline"] = cpu_baseline(wl, args.cpu_sample_s, kind)
    print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def run_update_scale(args, wl):
    """UpdateGradScale of Algorithm 1 alone, element-wise, over the whole parameter set:
    s = min(|g_small / (g_large + eps)|, s_max) with g_small = replica 1, g_large = replica 0
    (12 bytes per parameter).  One process; a diagnostic of k_scale_elem, not a step."""
    import torch

    from paper_2603_18112_gb300 import build as B
    from paper_2603_18112_gb300 import tula_ags as T
    from paper_2603_18112_gb300 import workloads as W
    if _dist()[0] > 1:
        raise SystemExit("--step-kind update-scale runs on one GPU")
    if not B.LIB.exists():
        B.build()
    T.lib()
    K = max(2, wl.K)
    buf = W.allocate(wl, "cuda", K=K)
    W.fill_grads(buf, wl, step=1)
    out = [torch.empty_like(t) for t in buf.w]
    hp = T.tula_ags_default_hparams(K)
    hp.granularity = T.TULA_SCALE_PER_ELEMENT
    keep = T._tensor_ptrs(out)
    hp.scale_elem = T.ctypes.cast(keep, T.c_void_p).value
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    # marshalled once, as a training loop would keep them (the binding's per-call marshalling
    # of 2 x n pointers costs more than the kernel on small sets)
    n = wl.pset.n_tensors
    g_small, g_large = T._tensor_ptrs(buf.g[1]), T._tensor_ptrs(buf.g[0])
    numels, sp = T._numels(buf.g[0]), T._stream_ptr(stream)
    lib = T.lib()

    def call():
        rc = lib.tula_ags_update_scale(g_small, g_large, numels, n, T.ctypes.byref(hp), sp)
        if rc:
            raise T.TulaError(rc, "tula_ags_update_scale")

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            call()
    stream.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    launches0 = T.tula_ags_launch_count()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            call()
        t1.record(stream)
    stream.synchronize()
    clocks = sampler.stop()
    ms = t0.elapsed_time(t1) / args.steps
    N = wl.pset.n_params
    peak, peak_kind = _peaks()
    gbs = scale_elem_bytes_per_param() * N / (ms / 1e3) / 1e9
    print(json.dumps({
        "metric": METRIC, "value": N / (ms / 1e3), "unit": UNIT, "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": _config(wl, wl.pset, "update-scale"),
        "roofline": {"bound": "hbm", "kernel": "k_scale_elem (UpdateGradScale, element-wise)",
                     "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                     "peak_kind": peak_kind, "traffic": _ncu_traffic("k_scale_elem", wl.name, N),
                     "bytes_per_launch": scale_elem_bytes_per_param() * N, "ms_per_launch": ms},
        "e2e": None, "gpu_launches": T.tula_ags_launch_count() - launches0, "clocks": clocks,
    }), flush=True)


def run_sharded(args, wl):
    """An Algorithm 1 step sharded over two ranks, emulated on one GPU by running the shards one
    after the other: tula_ags_shard_reduce on each half of the tensors, their shares of |G|^2
    added as integers (the exchange), tula_ags_shard_update on each half.  One process; it
    measures what sharding adds to a step (two passes per shard, the exchange) on the same
    parameter set, not a multi-GPU rate."""
    import torch

    from paper_2603_18112_gb300 import build as B
    from paper_2603_18112_gb300 import tula_ags as T
    from paper_2603_18112_gb300 import workloads as W
    if _dist()[0] > 1:
        raise SystemExit("--step-kind sharded runs its ranks one after the other on one GPU")
    if not B.LIB.exists():
        B.build()
    T.lib()
    buf = W.allocate(wl, "cuda")
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    K, n = wl.K, buf.pset.n_tensors
    cut = n // 2 + 1
    ranks = [T.AGSOptimizerStep(buf.w[lo:hi], [buf.g[k][lo:hi] for k in range(K)],
                                buf.m[lo:hi], s_max=wl.smax)
             for lo, hi in ((0, cut), (cut, n))]
    shares = [r.new_g2_share() for r in ranks]
    total = torch.zeros_like(shares[0])
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()

    def one_step(refresh=False):
        for r, sh in zip(ranks, shares):
            r.shard_reduce(wl.momentum, sh, refresh_scale=refresh, stream=stream)
        torch.add(shares[0], shares[1], out=total)
        for r in ranks:
            r.shard_update(wl.lr, wl.momentum, wl.weight_decay, total, refresh_scale=refresh,
                           stream=stream)

    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            one_step(refresh=(i == 0 and K > 1))
    stream.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    launches0 = T.tula_ags_launch_count()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            one_step()
        t1.record(stream)
    stream.synchronize()
    clocks = sampler.stop()
    ms = t0.elapsed_time(t1) / args.steps
    N = buf.pset.n_params
    peak, peak_kind = _peaks()
    per = step_min_bytes_per_param(K, False)
    gbs = per * N / (ms / 1e3) / 1e9
    config = _config(wl, buf.pset, "sharded")
    config["parallelism"] = "2 shards of whole tensors, run one after the other on one GPU"
    print(json.dumps({
        "metric": METRIC, "value": N / (ms / 1e3), "unit": UNIT, "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": config,
        "roofline": {"bound": "hbm", "kernel": "the whole sharded step (both shards)",
                     "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                     "peak_kind": peak_kind, "traffic": None,
                     "bytes_per_launch": per * N, "ms_per_launch": ms},
        "e2e": None, "gpu_launches": T.tula_ags_launch_count() - launches0, "clocks": clocks,
    }), flush=True)


def main():
    args = _args()
    from paper_2603_18112_gb300 import workloads as W
    wl = W.workload(args.workload)
    if args.impl == "reference":
        run_reference(args, wl)
    elif args.step_kind == "update-scale":
        run_update_scale(args, wl)
    elif args.step_kind == "sharded":
        run_sharded(args, wl)
    else:
        run_ours(args, wl)


if __name__ == "__main__":
    main()
