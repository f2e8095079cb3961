"""bench.py host logic on the CPU: the max-over-ranks timing reduction with
two gloo ranks, and the reference (oracle) arm's JSON line."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rank_main(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    bench.init_dist("gloo")
    bench.barrier()
    q.put((rank, bench.max_over_ranks(1.5 + rank)))
    import torch.distributed as dist
    dist.destroy_process_group()


def test_max_over_ranks_gloo_two_ranks():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + (os.getpid() % 1000)
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    assert got == [(0, 2.5), (1, 2.5)]


def test_reference_arm_prints_contract_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "single_256x512", "--steps", "2", "--warmup", "1"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "impl", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "cpu_baseline", "e2e", "config"):
        assert key in line
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0
    # one real step over the whole parameter set, reported as what ran
    assert line["steps"] == 1 and line["requested"] == {"steps": 2, "warmup": 1}
    assert abs(line["ms_per_step"] * line["value"] - 1e3) < 1e-6 * 1e3
    # the same config keys as the GPU arm's line
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_05088_gb300 import inputs
    want = dict(bench.workload_config(inputs.WORKLOADS["single_256x512"]), ns_schedule="auto")
    assert line["config"] == json.loads(json.dumps(want))


def test_reference_arm_nonzero_rank_is_silent():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "single_256x512", "--steps", "1"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert out.returncode == 0 and out.stdout.strip() == ""


def test_issued_flops_accounting():
    """Tensor-core flops issued per step: whole 256x256 tiles on and above
    the diagonal of the symmetric products, every tile of B X.  For a 256 x
    512 frame: Gram 1 tile x K 512, Poly 1 tile x K 256, B X 2 tiles x K 256."""
    from paper_2608_05088_gb300 import inputs
    one = inputs.Workload("t", 1, ((256, 512),), "f32", 1.0, 0.02, "malt", 1, ns_steps=1)
    t = 2.0 * 256 * 256
    assert one.ns_flops_issued() == t * (512 + 256 + 2 * 256)
    # with p a multiple of 256 the B X product is exact, the symmetric ones
    # carry the upper halves of the diagonal tiles on top of the minimum
    large = inputs.WORKLOADS["gpt2_large"]
    assert abs(large.ns_flops_issued() - 16.307453952e12) < 1e3
    assert large.ns_flops_min() < large.ns_flops_issued() < large.ns_flops_dense()



FAKE_SMI = r'''#!/usr/bin/env python3
# Stand-in for nvidia-smi's query loop: one timestamped row every 50 ms,
# 1700 MHz with the power cap active while the flag file exists ("load"),
# 2070 MHz otherwise.
import datetime, os, sys, time
flag = os.environ["FAKE_SMI_FLAG"]
while True:
    busy = os.path.exists(flag)
    stamp = datetime.datetime.now().strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    cap = "Active" if busy else "Not Active"
    sys.stdout.write(f"{stamp}, 0, {1700 if busy else 2070}, 2070, 900.0, 0x4, Not Active, "
                     f"Not Active, Not Active, {cap}\n")
    sys.stdout.flush()
    time.sleep(0.05)
'''


def _row(t, mhz, cap):
    import datetime
    stamp = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    return [stamp, "0", str(mhz), "2070", "900.0", "0x4", "Not Active", "Not Active",
            "Not Active", cap]


def test_clock_sampler_keeps_the_timed_region(tmp_path, monkeypatch):
    """Against a fake nvidia-smi: the clocks summary takes the samples dated
    inside begin() .. end(), not the idle ones before and after it."""
    import time
    sys.path.insert(0, ROOT)
    import bench
    smi = tmp_path / "nvidia-smi"
    smi.write_text(FAKE_SMI)
    smi.chmod(0o755)
    flag = tmp_path / "busy"
    monkeypatch.setenv("PATH", f"{tmp_path}{os.pathsep}{os.environ['PATH']}")
    monkeypatch.setenv("FAKE_SMI_FLAG", str(flag))
    s = bench.ClockSampler(0)
    s.start()
    flag.write_text("")
    s.begin()
    time.sleep(0.6)
    s.end()
    flag.unlink()
    out = s.stop()
    assert out["window"] == "timed region"
    assert out["sm_mhz"] == 1700 and out["reasons"] == ["sw_power_cap"]
    assert out["sm_max_mhz"] == 2070
    assert out["samples"] >= 5 and out["samples_total"] > out["samples"]


def test_clock_summary_fallbacks():
    sys.path.insert(0, ROOT)
    import bench
    t0 = 1.0e9
    rows = ([_row(t0 - 0.3 + 0.05 * i, 2070, "Not Active") for i in range(6)]
            + [_row(t0 + 0.05 * i, 1700, "Active") for i in range(1, 11)]
            + [_row(t0 + 0.6 + 0.05 * i, 2070, "Not Active") for i in range(6)])
    got = bench.ClockSampler.summarise(rows, t0, t0 + 0.55)
    assert (got["sm_mhz"], got["samples"], got["samples_total"]) == (1700, 10, 22)
    # a region shorter than the interval: the sample nearest its middle
    got = bench.ClockSampler.summarise(rows, t0 + 0.101, t0 + 0.109)
    assert got["samples"] == 1 and got["sm_mhz"] == 1700 and got["window"].startswith("nearest")
    # undated rows: every sample counts
    got = bench.ClockSampler.summarise([["n/a"] + r[1:] for r in rows], t0, t0 + 0.55)
    assert got["samples"] == 22 and got["window"].startswith("all samples")
    assert bench.ClockSampler.summarise([], t0, t0 + 1) is None


def test_roofline_traffic_holds_only_for_the_captured_kernel(tmp_path, monkeypatch):
    """roofline.traffic comes from an ncu summary only while every source the
    Newton-Schulz kernel compiles from is the one it was captured with; a
    changed source makes it null."""
    sys.path.insert(0, ROOT)
    import bench
    summary = tmp_path / "ncu.json"
    summary.write_text(json.dumps({"ns_sources_sha256": bench.ns_sources_sha256(),
                                   "dram_bytes_per_launch_full_size": 1.5e9}))
    monkeypatch.setattr(bench, "NCU_SUMMARY", str(summary))
    assert bench.ncu_traffic_per_launch(False) == 1.5e9
    assert bench.ncu_traffic_per_launch(True) is None          # no figure for that schedule
    changed = tmp_path / "common.cuh"
    changed.write_bytes(open(bench.NS_SOURCES[1], "rb").read() + b"// edited\n")
    monkeypatch.setattr(bench, "NS_SOURCES", [bench.NS_SOURCES[0], str(changed), bench.NS_SOURCES[2]])
    assert bench.ncu_traffic_per_launch(False) is None
