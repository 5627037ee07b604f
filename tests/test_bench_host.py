"""Host logic of bench.py: the replica aggregation across ranks (gloo,
world size 2, on CPU), the JSON line of the reference arm, the clock
summary and the recorded-traffic check."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench
    mx = bench.reduce_max(float(rank + 1) * 10.0, world)
    sm = bench.reduce_sum(float(rank + 1), world)
    bench.barrier(world)
    q.put((rank, mx, sm))
    dist.destroy_process_group()


def test_replica_aggregation_gloo_two_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    assert got == [(0, 20.0, 3.0), (1, 20.0, 3.0)]     # max of the times, sum of the work


def test_reference_arm_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                          "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    r = json.loads(lines[0])
    assert r["impl"] == "reference" and r["unit"] == "nnz-updates/s" and r["value"] > 0
    assert r["cpu_baseline"]["kind"] == "oracle" and r["cpu_baseline"]["cores"] == 1
    assert r["e2e"]["h2d_bytes_per_step"] == 0 and r["e2e"]["value"] == r["value"]
    assert r["higher_is_better"] is True and r["steps"] == 2 and r["warmup"] == 1


def test_reference_arm_other_ranks_exit_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny"],
                         capture_output=True, text=True, timeout=120, cwd=ROOT, env=env)
    assert out.returncode == 0 and out.stdout.strip() == ""


def test_clock_summary_reads_samples_and_throttle_reasons(tmp_path):
    # nvidia-smi --format=csv,noheader,nounits rows as the sampler records them
    sys.path.insert(0, ROOT)
    import bench
    csv = tmp_path / "clocks.csv"
    csv.write_text("0, 2070, 2070, 450.10, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n"
                   "0, 1995, 2070, 1399.70, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n"
                   "0, 2070, 2070, 600.00, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n"
                   "garbled line\n")

    class _File:
        name = str(csv)

    smp = bench.ClockSampler.__new__(bench.ClockSampler)
    smp.gpu, smp.proc, smp.file = "0", object(), _File()
    s = smp.summary()
    assert s["samples"] == 3 and s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["power_w_max"] == 1399.7 and s["reasons"] == ["sw_power_cap"]


def test_recorded_traffic_only_while_the_sources_match(tmp_path, monkeypatch):
    # the committed ncu traffic is reported only while the kernel's sources
    # hash as they did when it was captured, scaled to the run's nonzeros
    sys.path.insert(0, ROOT)
    import hashlib
    import bench
    csrc = tmp_path / "paper_1508_00703_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "window.cu").write_text("kernel A\n")
    (csrc / "common.cuh").write_text("helpers\n")
    (tmp_path / "profiles").mkdir()
    h = hashlib.sha256(b"kernel A\n" + b"helpers\n").hexdigest()
    (tmp_path / "profiles" / "k_sgd_window_low-conflict.md").write_text(
        f"traffic_bytes_per_launch: 123456\ntraffic_nnz: 1000\nsource_sha256: {h}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.recorded_traffic("k_sgd_window", "low-conflict", 1000) == 123456.0
    assert bench.recorded_traffic("k_sgd_window", "low-conflict", 100) == 12345.6
    (csrc / "window.cu").write_text("kernel B\n")
    assert bench.recorded_traffic("k_sgd_window", "low-conflict", 1000) is None
    assert bench.recorded_traffic("k_sgd_window", "zipf-1m", 1000) is None
