"""The benchmark's multi-rank path on CPU (gloo, world size 2).

With N GPUs every rank runs its own independent replica set (weak scaling);
the ranks exchange nothing but their timings.  These tests run that logic
with two gloo processes: the job time is the slowest rank's, the rate
counts every rank's units, and the reference arm runs on rank 0 only.
"""
import json
import os
import socket
import statistics
import subprocess
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, lr = bench.rank_env()
        assert (r, w, lr) == (rank, world, rank)
        dist.barrier()
        slowest = bench.max_over_ranks(1.5 + rank, dist, "cpu")    # rank 1 is slower
        out.put((rank, slowest, bench.job_rate(100.0, w, slowest)))
    finally:
        dist.destroy_process_group()


def test_timing_reduction_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.5, 2.5]
    assert [r[2] for r in res] == [80.0, 80.0]          # 2 ranks x 100 units / 2.5 s


def test_single_process_helpers():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.0) == 3.0
    assert bench.job_rate(10.0, 1, 2.0) == 5.0


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "0"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_reference_arm_json_line():
    """The reference arm (the oracle on the host cores) prints one JSON line
    with the contract's keys: the same metric and workload as the device
    arm, a cpu_baseline describing the run, and an e2e of its own value with
    no host-device traffic."""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["vs_baseline"] is None and d["data"] == "synthetic"
    assert d["config"]["workload"] == "decoder_1b"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    assert cb["cores"] == len(os.sched_getaffinity(0))          # every host core
    # ms_per_step is the measured time of a step of the sample, which ran:
    # well below a minute, not a full-size round extrapolated from it
    assert 0 < d["ms_per_step"] < 60e3
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_step_kernel_traffic_gate(tmp_path, monkeypatch):
    """bench.py reports the committed DRAM traffic only for the kernel
    instance and the kernel source it was captured from, scaled by the
    elements of the launch it times."""
    sys.path.insert(0, ROOT)
    import bench
    name = bench.step_kernel_name({"base": "adam", "n_mom": 3, "clip_mode": "none"}, "f32")
    assert name == "step_kernel<0, 3, 0, 0>"
    assert bench.step_kernel_name({"base": "adopt", "n_mom": 2}, "bf16") == "step_kernel<1, 2, 1, 0>"
    rec = tmp_path / "traffic.txt"
    rec.write_text("# capture\nkernel=%s\nelements=1000\ndram_bytes=44000\nsource_sha=%s\n"
                   % (name, bench.source_sha()))
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(rec))
    assert bench.measured_traffic(name, 5000) == 220000
    assert bench.measured_traffic("step_kernel<1, 2, 1, 0>", 5000) is None
    rec.write_text("kernel=%s\nelements=1000\ndram_bytes=44000\nsource_sha=0000000000000000\n" % name)
    assert bench.measured_traffic(name, 5000) is None
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(tmp_path / "missing.txt"))
    assert bench.measured_traffic(name, 5000) is None



def test_clock_sample_summary():
    """The clocks record of the bench line: median SM clock under load,
    maximum clock, slowdown reasons seen active; idle and malformed samples
    do not count."""
    sys.path.insert(0, ROOT)
    import bench
    idle = "0, 1965, 2070, 180.5, 0x0000000000000001, Not Active, Not Active, Not Active, Not Active"
    busy = "0, 2070, 2070, 950.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active"
    capped = "0, 1890, 2070, 1390.2, 0x0000000000000004, Not Active, Not Active, Not Active, Active"
    slow = "0, 1500, 2070, 900.0, 0x0000000000000008, Active, Not Active, Not Active, Not Active"
    s = bench.parse_clock_samples([idle, busy, busy, "garbage", "0, [N/A], 2070, 1, x, a, b, c, d"])
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0 and s["reasons"] == []
    assert s["samples"] == 3 and s["power_w_max"] == 950.0
    s = bench.parse_clock_samples([busy, capped, capped, slow])
    assert s["reasons"] == ["hw_slowdown", "sw_power_cap"]
    assert s["sm_mhz"] == statistics.median([2070.0, 1890.0, 1890.0, 1500.0])
    assert bench.parse_clock_samples([])["reasons"] == ["no samples"]


def test_sweep_options(monkeypatch):
    """bench.py --sweep visits M in {1,2,4,8} and N in {1..4} unless told
    otherwise; --sweep-M / --sweep-N take other replica and momentum counts
    (the block-staged fused step's range, for instance)."""
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr("sys.argv", ["bench.py", "--sweep"])
    a = bench.parse_args()
    assert (a.sweep, a.sweep_M, a.sweep_N, a.sweep_log2n) == (True, "1,2,4,8", "1,2,3,4", "20,24,27,30")
    monkeypatch.setattr("sys.argv", ["bench.py", "--sweep", "--sweep-M", "9,16,64", "--sweep-N", "3",
                                     "--sweep-log2n", "26"])
    a = bench.parse_args()
    assert [int(v) for v in a.sweep_M.split(",")] == [9, 16, 64]
    assert (a.sweep_N, a.sweep_log2n) == ("3", "26")
