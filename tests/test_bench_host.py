"""Host-side logic of bench.py on the CPU: the trimmed mean of Eq. 3, workload
resizing, the traffic record's staleness check, the reference (oracle) arm,
and the multi-rank timing reduction over gloo with two ranks."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_trimmed_mean_matches_oracle():
    rng = np.random.default_rng(0)
    for R, k in ((30, 3), (7, 1), (5, 0), (100, 10)):
        t = list(rng.exponential(1.0, R))
        assert bench.trimmed_mean(t, k) == pytest.approx(oracle.trimmed_mean(t, k), rel=1e-15)
    with pytest.raises(ValueError):
        bench.trimmed_mean([1.0, 2.0], 1)


def test_workload_resize_keeps_dtype_and_names_it():
    from paper_2512_22147_gb300 import inputs

    class A:
        workload = "i32_4001x100003_lda100008"
        M, N, lda, batch = None, 25000, 25008, None

    w = bench.workload_from_args(inputs, A)
    assert (w.M, w.N, w.lda, w.dtype) == (4001, 25000, 25008, "i32")
    assert "resized" in w.name
    A.lda = None
    assert bench.workload_from_args(inputs, A).lda == 25000


def test_bytes_counted():
    from paper_2512_22147_gb300 import inputs
    w = inputs.WORKLOADS["f32_16384x16384"]
    assert w.bytes_counted() == 16384 * 16384 * 4 + 4 * 16384 * 4
    w = inputs.WORKLOADS["i32_4001x100003_lda100008"]
    assert w.bytes_counted() == 4001 * 100003 * 4 + (4001 + 100003) * (4 + 8)


def test_traffic_record_goes_stale_with_the_kernel(tmp_path, monkeypatch):
    rec = {"wl": {"kernel_source_hash": bench.kernel_source_hash(),
                  "dram_bytes_per_launch": 123}}
    f = tmp_path / "traffic.json"
    f.write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(f))
    assert bench.recorded_traffic("wl") == 123
    assert bench.recorded_traffic("other") is None
    rec["wl"]["kernel_source_hash"] = "0" * 16
    f.write_text(json.dumps(rec))
    assert bench.recorded_traffic("wl") is None


def test_reference_arm_prints_one_json_line():
    out = subprocess.run(
        [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
         "--workload", "f32_1024x1024", "--steps", "3", "--warmup", "3",
         "--cpu-seconds", "0.5"], capture_output=True, text=True, check=True, cwd=ROOT)
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "GB/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0


def test_reference_arm_other_ranks_stay_silent():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    out = subprocess.run(
        [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
         "--workload", "f32_1024x1024", "--steps", "3", "--warmup", "3"],
        capture_output=True, text=True, check=True, cwd=ROOT, env=env)
    assert out.stdout.strip() == ""


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        got = bench.max_over_ranks(torch, 10.0 + rank * 5.0, world, torch.device("cpu"))
        q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_with_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    assert res == [(0, 15.0), (1, 15.0)]
