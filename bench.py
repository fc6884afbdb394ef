"""Benchmark of the MT-DAO hot path on GB300.

One benchmark "step" is one communication round of the workload: H local
optimizer steps of all M replicas (H = the largest sync period), the round's
due replica averages fused into its last step.  Default workload: the ~1B
decoder-shaped parameter list (1,311,086,592 fp32 per replica, M=4, N=3,
Adam, H=32), the configuration the bandwidth target is quoted on.

Printed (rank 0, one JSON line): params/s = M * n * H / round time (whole
job, all ranks), plus the roofline of the dominant kernel (the local-step
kernel, timed per launch with CUDA events on its stream), the standalone
sync kernel's bandwidth, an end-to-end figure through the host-buffer C-ABI
call, and the CPU oracle timed on a bounded sample (one core and all the
host's cores).  The default run also times the ~350M decoder list (ADOPT,
bf16 gradients, M = 8, per-state periods K_x = 64, K_u = K_v = 16) in a
child process and reports it under "workloads".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload decoder_1b|gpt2_small|decoder_350m|tiny]
For N > 1 (torchrun) every rank runs its own independent replica set
(weak scaling); only the timing is reduced across ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from synth import workloads as W  # noqa: E402

PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "step_kernel_traffic.txt")
STEP_KERNEL_SRC = os.path.join(ROOT, "paper_2510_05361_gb300", "csrc", "step_kernels.cuh")
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0    # vendor figure for GB300 HBM3e, for context beside the measured peak
L2_BYTES = 129 * 2 ** 20
SOLO_LAUNCHES = 20          # timed launches of each standalone kernel (after 2 untimed)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="decoder_1b", choices=sorted(W.WORKLOADS))
    ap.add_argument("--e2e-rounds", type=int, default=2)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="flat-vector sweep: one JSON line per (n, M, N) with step, fused "
                         "step+sync and sync bandwidth, and the round rate for H in {1, 8, 64}")
    ap.add_argument("--sweep-log2n", default="20,24,27,30")
    ap.add_argument("--sweep-M", default="1,2,4,8", help="replica counts of the sweep")
    ap.add_argument("--sweep-N", default="1,2,3,4", help="momentum counts of the sweep")
    ap.add_argument("--second-workload", default="decoder_350m",
                    help="workload timed in a child process after the main one ('' = none)")
    return ap.parse_args()


def rank_env():
    """(rank, world size, local rank) from the torchrun environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(value: float, dist=None, device="cpu") -> float:
    """The largest value over all ranks (a job takes as long as its slowest
    rank); the identity without a process group."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput: every rank processes its own units (weak
    scaling, no data-path collective), in the slowest rank's time."""
    return world * units_per_rank / seconds


def round_len(opt) -> int:
    periods = [opt["period_x"], opt.get("period_v", 0)] + list(opt["period_u"])
    return max(p for p in periods if p > 0)


def hbm_peak():
    try:
        with open(PEAKS_FILE) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def source_sha() -> str:
    with open(STEP_KERNEL_SRC, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def step_kernel_name(opt: dict, grad_dtype: str) -> str:
    """Template instance of the plain step kernel a workload launches."""
    base = {"adam": 0, "adopt": 1, "sgdm": 2}[opt["base"]]
    clip = 1 if opt.get("clip_mode") == "global_norm" else 0
    return "step_kernel<%d, %d, %d, %d>" % (base, opt["n_mom"], 1 if grad_dtype == "bf16" else 0, clip)


def measured_traffic(kernel: str, per_launch_units: int):
    """DRAM bytes per launch of the step kernel from the committed ncu
    summary, scaled by elements to this launch; None if absent, if it was
    taken on another template instance, or if the kernel source changed
    since the capture."""
    rec = {}
    try:
        with open(TRAFFIC_FILE) as f:
            for line in f:
                line = line.strip()
                if line and not line.startswith("#") and "=" in line:
                    k, v = line.split("=", 1)
                    rec[k] = v
        if rec.get("source_sha") != source_sha() or rec.get("kernel") != kernel:
            return None
        per_unit = float(rec["dram_bytes"]) / float(rec["elements"])
    except Exception:
        return None
    return int(round(per_unit * per_launch_units))


# --------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.close()
        with open(self.path) as f:
            summary = parse_clock_samples(f)
        os.unlink(self.path)
        return summary


def parse_clock_samples(lines) -> dict:
    """Summary of nvidia-smi samples in ClockSampler.FIELDS order (csv,
    no header, no units): the median SM clock over the samples drawn under
    load (power above half the maximum seen), the maximum clock, and every
    slowdown reason seen active."""
    sm, smax, reasons, power = [], [], set(), []
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for line in lines:
        parts = [p.strip() for p in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            smax.append(float(parts[2]))
            power.append(float(parts[3]))
        except ValueError:
            continue
        for name, val in zip(names, parts[5:9]):
            if val.lower().startswith("active"):
                reasons.add(name)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
    loaded = [s for s, p in zip(sm, power) if p > 0.5 * max(power)] or sm
    return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax),
            "reasons": sorted(reasons), "samples": len(sm),
            "power_w_max": max(power)}


# --------------------------------------------------------------------- CPU oracle

def host_cores() -> int:
    """Host cores this process may run on."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


class OracleSlices:
    """The CPU oracle, as it stands, on `threads` disjoint slices of a
    workload's elements (n_per_thread consecutive elements of every replica
    each; slice k starts at element k * n_per_thread).  Each slice is its own
    oracle instance with all M replicas, run by its own thread (the oracle's
    C calls release the interpreter lock).  Without global-norm clipping the
    elements of the method are independent, so the slices together compute
    exactly what one oracle over all of them would; nothing in the oracle is
    changed or tuned for this."""

    def __init__(self, w, n_per_thread: int, threads: int):
        import concurrent.futures as cf

        import numpy as np

        from oracle.oracle import Oracle
        from synth import generators as G

        assert w["opt"].get("clip_mode", "none") != "global_norm", \
            "global-norm clipping couples the elements of a replica"
        self.w, self.opt, self.M = w, w["opt"], w["M"]
        self.H = round_len(self.opt)
        self.n_per, self.threads = n_per_thread, threads
        lay = W.layout(w["shapes"])
        self.slices = []
        for k in range(threads):
            idx = np.arange(k * n_per_thread, (k + 1) * n_per_thread, dtype=np.int64)
            x0 = G.init_params(w, lay, W.INIT_SEED, idx).astype(np.float64)
            g = np.stack([G.grads(w, lay, W.GRAD_SEED, m, 0, idx) for m in range(self.M)]).astype(np.float64)
            self.slices.append((Oracle(self.opt, self.M, n_per_thread, x0=x0), g))
        self.pool = cf.ThreadPoolExecutor(max_workers=threads)
        self.t = 0

    def round(self) -> float:
        """One round (H local steps of every slice, all replicas); returns
        its wall time in seconds.  The oracle performs a round's averages
        at the start of the next round's first step (Algorithm 1's form)."""
        t, H, lr = self.t, self.H, self.opt["lr"]

        def work(item):
            o, g = item
            for s in range(H):
                o.step(t + s, lr, g)

        t0 = time.perf_counter()
        list(self.pool.map(work, self.slices))
        dt = time.perf_counter() - t0
        self.t += H
        return dt

    def units_per_round(self) -> int:
        return self.M * self.n_per * self.threads * self.H

    def describe(self) -> str:
        return ("%d thread(s) x %d elements of every replica (M = %d, elements [0, %d) of the "
                "workload) x rounds of %d local steps with their averages; one resident gradient "
                "batch" % (self.threads, self.n_per, self.M, self.threads * self.n_per, self.H))

    def close(self):
        self.pool.shutdown()


def cpu_baseline(w) -> dict:
    """The oracle timed on the host: one round on one core (2^21 elements
    of every replica, ~13 s on a Grace core) and one round on every core
    (2^19 elements per core)."""
    one = OracleSlices(w, 1 << 21, 1)
    s1 = one.round()
    r1 = one.units_per_round() / s1
    d1 = one.describe()
    one.close()
    del one
    cores = host_cores()
    allc = OracleSlices(w, 1 << 19, cores)
    sa = allc.round()
    ra = allc.units_per_round() / sa
    da = allc.describe()
    allc.close()
    return {"value": ra, "unit": "params/s", "cores": cores, "kind": "oracle", "sample": da,
            "seconds": round(sa, 2),
            "one_core": {"value": r1, "unit": "params/s", "cores": 1, "sample": d1, "seconds": round(s1, 2)}}


def run_reference(args):
    rank, _, _ = rank_env()
    if rank != 0:
        return 0
    w = W.get(args.workload)
    cores = host_cores()
    sl = OracleSlices(w, 1 << 18, cores)
    for _ in range(max(args.warmup, 0)):
        sl.round()
    secs = [sl.round() for _ in range(args.steps)]
    sl.close()
    med = statistics.median(secs)
    value = sl.units_per_round() / med
    desc = sl.describe()
    line = {
        "impl": "reference",
        "metric": "fused MT-DAO step params/s (replica-parameter updates per second, syncs included)",
        "value": value,
        "unit": "params/s",
        "n_gpus": args.gpus,
        "steps": args.steps,
        "warmup": args.warmup,
        # measured: one step = one round of the bounded sample below (not the
        # full workload, which the oracle would take hours for)
        "ms_per_step": 1e3 * med,
        "ms_per_step_measured_on": "the sample (%d replica-element updates per round)" % sl.units_per_round(),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w["name"], "desc": w["desc"], "sample": desc},
        "cpu_baseline": {"value": value, "unit": "params/s", "cores": cores, "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": "params/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------- GPU arm

def run_ours(args):
    import torch

    import paper_2510_05361_gb300 as P
    from synth.device import DeviceInputs

    rank, world, local = rank_env()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    P.load()

    w = W.get(args.workload)
    opt, M = w["opt"], w["M"]
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    H = round_len(opt)
    gdt = P.BF16 if w["grad_dtype"] == "bf16" else P.F32
    g_bytes = 2 if gdt == P.BF16 else 4
    n_states = 1 + opt["n_mom"] + (0 if opt["base"] == "sgdm" else 1)
    step_bytes = W.bytes_per_step(w)
    stream = torch.cuda.current_stream()

    eng = P.MTDAO(opt, M, w["shapes"], stream=stream.cuda_stream)
    inputs = DeviceInputs(w, lay, W.GRAD_SEED, W.INIT_SEED)
    eng.set_params(inputs.init_params())
    grads = inputs.grads(0)            # one resident batch, reused every local step
    torch.cuda.synchronize()

    small = step_bytes < 8 * L2_BYTES
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda") if small else None

    masks = []

    def one_round(events=None):
        for k in range(H):
            mask = eng.sync_due()
            if flush is not None:
                flush.fill_(1.0)
            if events is not None:
                events[k][0].record(stream)
                masks.append(mask)
            P.mtdao_step(eng.h, grads.data_ptr(), gdt, opt["lr"], mask)
            if events is not None:
                events[k][1].record(stream)

    for _ in range(args.warmup):
        one_round()
    torch.cuda.synchronize()

    sampler = ClockSampler(local)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)
    rounds_ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(H)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for r in range(args.steps):
        one_round(rounds_ev[r])
    end.record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    clocks = sampler.stop()
    elapsed_ms = start.elapsed_time(end)
    launch_ms = [[a.elapsed_time(b) for a, b in rnd] for rnd in rounds_ev]
    flat = [ms for rnd in launch_ms for ms in rnd]
    plain = [ms for ms, mk in zip(flat, masks) if mk == 0]
    sync_steps = [ms for ms, mk in zip(flat, masks) if mk != 0]
    if small:
        # L2 was flushed before every launch; time only the launches.
        elapsed_ms = sum(ms for rnd in launch_ms for ms in rnd)
    elapsed_ms = max_over_ranks(elapsed_ms, dist, "cuda")
    value = job_rate(M * n * H * args.steps, world, elapsed_ms / 1e3)
    step_ms = statistics.mean(plain)
    peak, peak_kind = hbm_peak()
    achieved = step_bytes / (step_ms / 1e3) / 1e9

    def launches(fn, reps=SOLO_LAUNCHES, skip=2):
        """Device times (ms) of `reps` launches of fn after `skip` untimed
        ones, each bracketed by events on the launching stream."""
        out = []
        for i in range(skip + reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            if flush is not None:
                flush.fill_(1.0)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            if i >= skip:
                out.append(a.elapsed_time(b))
        return out

    # standalone replica-average kernel (all states), timed separately
    all_mask = (1 << n_states) - 1
    sync_ms = launches(lambda: P.mtdao_sync(eng.h, all_mask))
    sync_bytes = W.bytes_per_sync(w, n_states)
    sync_gbs = sync_bytes / (statistics.median(sync_ms) / 1e3) / 1e9

    # the same average with the cross-worker diagnostics formed in its pass
    stats_out = torch.empty((n_states, 2 + 2 * M), dtype=torch.float64, device="cuda")
    stats_ms = launches(lambda: P.mtdao_sync_stats(eng.h, all_mask, stats_out.data_ptr()))

    # pseudo-gradient diagnostics: a read-only pass over x and the anchor
    P.mtdao_track_anchor(eng.h, 1)
    pg_out = torch.empty((2 * M + 2,), dtype=torch.float64, device="cuda")
    pg_ms = launches(lambda: P.mtdao_pseudo_grad_stats(eng.h, 0, pg_out.data_ptr()))
    P.mtdao_track_anchor(eng.h, 0)
    pg_bytes = (M + 1) * n * 4

    # S0: per-replica gradient sum of squares (the clip(g, rho) pre-pass) and
    # the non-finite count, each one read of the resident gradients
    norm_out = torch.empty((M,), dtype=torch.float64, device="cuda")
    norm_ms = launches(lambda: P.mtdao_grad_sqnorm(eng.h, grads.data_ptr(), gdt, norm_out.data_ptr()))
    nonfinite_ms = launches(lambda: P.mtdao_grad_nonfinite(eng.h, grads.data_ptr(), gdt, norm_out.data_ptr()))
    grad_bytes = M * n * g_bytes

    # end to end through the host-buffer C-ABI call
    e2e = None
    if not args.no_e2e and args.e2e_rounds > 0:
        host_mem = "pinned"
        try:
            host_g = torch.empty((M, n), dtype=grads.dtype, pin_memory=True)
        except RuntimeError:
            # many ranks pinning tens of GB each can exhaust pinnable memory:
            # pageable gradients go through the library's staging copy
            host_g = torch.empty((M, n), dtype=grads.dtype)
            host_mem = "pageable"
        host_g.copy_(grads)
        host_x = torch.empty((n,), dtype=torch.float32, pin_memory=host_mem == "pinned")
        P.mtdao_step_host(eng.h, host_g.data_ptr(), gdt, opt["lr"], eng.sync_due())
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_rounds):
            for _ in range(H):
                P.mtdao_step_host(eng.h, host_g.data_ptr(), gdt, opt["lr"], eng.sync_due())
            P.mtdao_copy_state_to_host(eng.h, 0, 0, host_x.data_ptr())   # round's synced x
        torch.cuda.synchronize()
        e2e_s = max_over_ranks(time.perf_counter() - t0, dist, "cuda")
        e2e = {"value": job_rate(M * n * H * args.e2e_rounds, world, e2e_s), "unit": "params/s",
               "h2d_bytes_per_step": H * M * n * g_bytes, "d2h_bytes_per_step": n * 4,
               "rounds": args.e2e_rounds, "host_memory": host_mem}
        del host_g

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w)

    # the second named workload, in a fresh process (its allocations are
    # not the first ones after a large free, and it does not share this
    # process's state); this process keeps its memory meanwhile
    second = None
    if rank == 0 and world == 1 and args.second_workload and args.second_workload != w["name"]:
        second = run_child_workload(args.second_workload, args.steps, args.warmup)

    traffic = measured_traffic(step_kernel_name(opt, w["grad_dtype"]), M * n)
    line = {
        "metric": "fused MT-DAO step params/s (replica-parameter updates per second, syncs included)",
        "value": value,
        "unit": "params/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {
            "workload": w["name"], "desc": w["desc"], "M": M, "n_padded": n, "n_mom": opt["n_mom"],
            "base": opt["base"], "grad_dtype": w["grad_dtype"], "local_steps_per_step": H,
            "periods": {"x": opt["period_x"], "u": list(opt["period_u"]), "v": opt.get("period_v", 0)},
            "step": "one communication round: H local steps, the due averages fused into the last",
            "grads": "one resident synthetic gradient batch per replica, reused every local step",
            "l2": ("L2 flushed before every launch; time = sum of launch times" if small else
                   "inputs larger than L2 (%.0f GB resident)" % ((n_states * 4 + g_bytes) * M * n / 1e9)),
            "parallelism": "replicas only" if world == 1 else "independent replica set per GPU",
        },
        "step_kernel": {"ms_mean": step_ms, "ms_median": statistics.median(plain), "ms_min": min(plain),
                        "launches": len(plain), "bytes": step_bytes,
                        "gbs": achieved, "frac_of_nominal": achieved / NOMINAL_HBM_GBS,
                        "params_per_s": M * n / (step_ms / 1e3),
                        "model_params_per_s": n / (step_ms / 1e3)},
        "sync_step_kernel": {"ms_mean": statistics.mean(sync_steps),
                             "gbs": step_bytes / (statistics.mean(sync_steps) / 1e3) / 1e9,
                             "launches_per_round": len(sync_steps) // args.steps},
        "sync_kernel": {"ms_median": statistics.median(sync_ms), "ms_min": min(sync_ms),
                        "launches": len(sync_ms), "bytes": sync_bytes, "gbs": sync_gbs,
                        "frac_of_nominal": sync_gbs / NOMINAL_HBM_GBS,
                        "frac": sync_gbs / peak, "states": n_states},
        "sync_stats_kernel": ({"ms_median": statistics.median(stats_ms), "ms_min": min(stats_ms),
                               "gbs": sync_bytes / (statistics.median(stats_ms) / 1e3) / 1e9,
                               "frac": sync_bytes / (statistics.median(stats_ms) / 1e3) / 1e9 / peak}
                              if stats_ms else None),
        "pseudo_grad_stats_kernel": ({"ms_median": statistics.median(pg_ms), "ms_min": min(pg_ms),
                                      "bytes": pg_bytes,
                                      "gbs": pg_bytes / (statistics.median(pg_ms) / 1e3) / 1e9}
                                     if pg_ms else None),
        "grad_sqnorm_kernel": {"ms_median": statistics.median(norm_ms), "ms_min": min(norm_ms),
                               "bytes": grad_bytes,
                               "gbs": grad_bytes / (statistics.median(norm_ms) / 1e3) / 1e9,
                               "frac": grad_bytes / (statistics.median(norm_ms) / 1e3) / 1e9 / peak},
        "grad_nonfinite_kernel": {"ms_median": statistics.median(nonfinite_ms), "bytes": grad_bytes,
                                  "gbs": grad_bytes / (statistics.median(nonfinite_ms) / 1e3) / 1e9},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
                     "kernel": step_kernel_name(opt, w["grad_dtype"])},
        "cpu_baseline": cpu,
        "workloads": second,
        "e2e": e2e,
        "gpu_launches": args.steps * H * (3 if opt.get("clip_mode") == "global_norm" else 1),
        "clocks": clocks,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    eng.close()
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_child_workload(name: str, steps: int, warmup: int):
    """Run this benchmark on workload `name` in a child process (no e2e, no
    CPU baseline) and summarise its kernel and round figures."""
    cmd = [sys.executable, os.path.abspath(__file__), "--workload", name, "--steps", str(steps),
           "--warmup", str(warmup), "--no-e2e", "--no-cpu-baseline", "--second-workload", ""]
    env = {k: v for k, v in os.environ.items()
           if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK", "LOCAL_WORLD_SIZE", "MASTER_ADDR", "MASTER_PORT")}
    try:
        r = subprocess.run(cmd, capture_output=True, text=True, timeout=900, env=env, cwd=ROOT)
    except subprocess.TimeoutExpired:
        return {name: {"error": "timed out"}}
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    if r.returncode != 0 or not lines:
        return {name: {"error": "exit %d: %s" % (r.returncode, r.stderr.strip().splitlines()[-1:])}}
    c = json.loads(lines[-1])
    cfg = c["config"]
    return {name: {
        "value": c["value"], "unit": c["unit"], "ms_per_step": c["ms_per_step"],
        "step": cfg["step"], "local_steps_per_step": cfg["local_steps_per_step"],
        "M": cfg["M"], "n_padded": cfg["n_padded"], "n_mom": cfg["n_mom"], "base": cfg["base"],
        "grad_dtype": cfg["grad_dtype"], "periods": cfg.get("periods"),
        "step_kernel": {k: c["step_kernel"][k] for k in ("ms_mean", "ms_median", "gbs", "bytes")},
        "step_kernel_frac": c["roofline"]["frac"],
        "sync_step_kernel": c["sync_step_kernel"],
        "sync_kernel": {k: c["sync_kernel"][k] for k in ("ms_median", "gbs", "frac", "states")},
        "sync_stats_kernel": c.get("sync_stats_kernel"),
        "pseudo_grad_stats_kernel": c.get("pseudo_grad_stats_kernel"),
        "grad_sqnorm_kernel": c.get("grad_sqnorm_kernel"),
        "peak": c["roofline"]["peak"], "kernel": c["roofline"]["kernel"],
        "gpu_launches": c["gpu_launches"], "clocks": c["clocks"],
    }}


def run_sweep(args):
    """Flat fp32 vector n = 2^k, M in --sweep-M (default {1,2,4,8}), N in
    --sweep-N (default {1..4}) (Adam, f32 gradients).  Each (n, M, N) point times 6 launches (2 warm-up) of the
    plain step, the fused step + average of every state, and the standalone
    average; per H in {1, 8, 64} a round is (H-1) plain steps and one fused
    step, so its rate follows from those times."""
    import torch

    import paper_2510_05361_gb300 as P
    from synth.device import DeviceInputs

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    P.load()
    peak, peak_kind = hbm_peak()
    stream = torch.cuda.current_stream()

    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_on = [False]

    def timed(fn, reps=6, skip=2):
        out = []
        for i in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            if flush_on[0]:
                flush.fill_(1.0)          # evict the previous launch's data from L2
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            if i >= skip:
                out.append(a.elapsed_time(b))
        return statistics.median(out)

    for k in [int(v) for v in args.sweep_log2n.split(",")]:
        for M in [int(v) for v in args.sweep_M.split(",")]:
            for N in [int(v) for v in args.sweep_N.split(",")]:
                w = W.sweep_point(k, M, N, 8)
                n_states = N + 2
                need = M * (1 << k) * (4 * n_states + 4) + (4 << 30)
                free = torch.cuda.mem_get_info()[0]
                rec = {"sweep": True, "log2_n": k, "M": M, "N": N, "base": "adam", "grad_dtype": "f32"}
                if need > free:
                    rec["skipped"] = "needs %.0f GB, %.0f GB free" % (need / 1e9, free / 1e9)
                    print(json.dumps(rec), flush=True)
                    continue
                lay = W.layout(w["shapes"])
                eng = P.MTDAO(w["opt"], M, w["shapes"], stream=stream.cuda_stream)
                inputs = DeviceInputs(w, lay, W.GRAD_SEED, W.INIT_SEED)
                eng.set_params(inputs.init_params())
                g = inputs.grads(0)
                all_mask = (1 << n_states) - 1
                lr = w["opt"]["lr"]
                flush_on[0] = W.bytes_per_step(w) < 8 * L2_BYTES
                rec["l2_flushed"] = flush_on[0]
                t_step = timed(lambda: P.mtdao_step(eng.h, g.data_ptr(), P.F32, lr, 0))
                t_fused = timed(lambda: P.mtdao_step(eng.h, g.data_ptr(), P.F32, lr, all_mask))
                t_sync = timed(lambda: P.mtdao_sync(eng.h, all_mask)) if M > 1 else None
                step_bytes = W.bytes_per_step(w)
                sync_bytes = W.bytes_per_sync(w, n_states)
                rec.update({
                    "step_ms": t_step, "step_gbs": step_bytes / t_step / 1e6,
                    "step_frac": step_bytes / t_step / 1e6 / peak,
                    "fused_ms": t_fused, "fused_gbs": step_bytes / t_fused / 1e6,
                    "fused_frac": step_bytes / t_fused / 1e6 / peak,
                    "sync_ms": t_sync,
                    "sync_gbs": (sync_bytes / t_sync / 1e6) if t_sync else None,
                    "sync_frac": (sync_bytes / t_sync / 1e6 / peak) if t_sync else None,
                    "peak_gbs": peak, "peak_kind": peak_kind,
                    "round_params_per_s": {
                        str(H): M * lay["n_padded"] * H / (((H - 1) * t_step + t_fused) / 1e3)
                        for H in (1, 8, 64)},
                })
                print(json.dumps(rec), flush=True)
                del g
                eng.close()
                torch.cuda.empty_cache()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
