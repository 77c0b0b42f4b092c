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
    name = "dmv::dualmv_stream_kernel<float, 8, 4, 6, 1, 0, 3, 0>"
    rec = {"wl": {"kernel_source_hash": bench.kernel_source_hash("dualmv_stream_kernel"),
                  "kernel": name, "dram_bytes_per_launch": 123}}
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
    # The native arm's config for the same workload: the same dict (its L2
    # line as the native arm decides it, a flush for this 4 MiB workload).
    from paper_2512_22147_gb300 import inputs
    w = inputs.WORKLOADS["f32_1024x1024"]
    assert d["config"] == bench.workload_config(w, w.bytes_counted(), True, 1)
    big = inputs.WORKLOADS["f32_16384x16384"]
    cfg = bench.workload_config(big, big.bytes_counted(), False, 1)
    assert cfg["op"] == "bicg" and cfg["bytes_per_step"] == big.bytes_counted()
    assert "larger than L2" in cfg["l2"]


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


def test_launch_list_parser_and_traffic_record(tmp_path, monkeypatch):
    """The ncu CSV parser groups metric rows by launch, converts units, and
    the traffic record keeps the streaming kernel's bytes per launch."""
    hdr = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream",'
           '"Block Size","Grid Size","Device","CC","Section Name","Metric Name","Metric Unit",'
           '"Metric Value"\n')

    def row(i, name, metric, unit, val):
        return (f'"{i}","1","python3","h","{name}","1","7","(288, 1, 1)","(152, 1, 1)","0",'
                f'"10.3","Command line profiler metrics","{metric}","{unit}","{val}"\n')

    k = "void dmv::dualmv_stream_kernel<float, 8, 4, 6, 1, 0>(dmv::Params<float>)"
    c = "void dmv::dualmv_combine_kernel<float>(dmv::Params<float>, int, int)"
    lines = ["==PROF== Connected to process 1\n", hdr]
    for i, (name, us, mb) in enumerate([(k, 160.0, 1000.0), (c, 8.0, 4.0), (k, 170.0, 1002.0)]):
        lines += [row(i, name, "dram__bytes_read.sum", "Mbyte", f"{mb:.1f}"),
                  row(i, name, "dram__bytes_write.sum", "Kbyte", "500"),
                  row(i, name, "gpu__time_duration.sum", "ns", f"{us * 1e3:.0f}")]
    csv_path = tmp_path / "launches.csv"
    csv_path.write_text("".join(lines))
    parsed = bench.parse_launch_list(str(csv_path))
    assert [p[0] for p in parsed] == [0, 1, 2]
    assert parsed[0][2]["dram__bytes_read.sum"] == 1000e6
    assert parsed[0][2]["dram__bytes_write.sum"] == 500e3
    md = bench.summarize_launches(str(csv_path), "cmd")
    assert "| `dmv::dualmv_stream_kernel<float, 8, 4, 6, 1, 0>` | 2 | 330.0 | 97.6 % |" in md
    rec = tmp_path / "traffic.json"
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(rec))
    # A small-case capture scaled to the full workload (here 4x its bytes).
    md = bench.record_traffic(str(csv_path), "wl", "cmd", full_bytes=4000, case_bytes=1000,
                              case="a small case")
    full = int(round(4 * (1001e6 + 500e3)))
    assert "scaled to the full workload" in md
    assert bench.recorded_traffic("wl") == full
    assert bench.recorded_traffic("wl", "dualmv_stream_kernel", (8, 4, 6)) == full
    assert bench.recorded_traffic("wl", "dualmv_stream_kernel", (8, 4, 4)) is None
    assert bench.recorded_traffic("wl", "dualmv_wide_i32_kernel", (8, 4, 6)) is None
    # Batched calls name the family only (their default kernel has no variant).
    assert bench.recorded_traffic("wl", "dualmv_stream_kernel", None) == full
    assert bench.recorded_traffic("wl", "dualmv_wide_i32_kernel", None) is None
    assert bench.recorded_traffic("other") is None
    assert bench.kernel_shape("dmv::dualmv_stream_f64e_kernel<8, 4, 3, 256, 0, 3, 2, 1>") == \
        (8, 4, 3)
    assert bench.kernel_shape("dmv::dualmv_wide_i32_kernel<8, 8, 3>") == (8, 8, 3)
    assert bench.kernel_shape("dmv::dualmv_small_cluster_kernel<8, 3>") == (8, 3)
    assert bench.kernel_family("void dmv::dualmv_small_cluster_kernel<8, 3>") in \
        bench.KERNEL_FAMILIES


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_sample_parity_accepts_oracle_and_rejects_a_perturbation(dtype):
    """The bench's parity block: the oracle's own outputs pass; one output
    moved by far more than the bar fails."""
    import oracle
    from paper_2512_22147_gb300 import inputs
    w = inputs.Workload("t", dtype, 40, 70, 72, {"f32": "uniform", "f64": "normal",
                                                 "i32": "int8"}[dtype], 3)
    A, p, r = inputs.generate(w)
    A_np, p_np, r_np = A.numpy(), p.numpy(), r.numpy()
    q_o, s_o = oracle.dualmv(A_np, p_np, r_np, N=w.N)
    cast = {"f32": np.float32, "f64": np.float64, "i32": np.int64}[dtype]
    qg, sg = q_o.astype(cast), s_o.astype(cast)
    ok = bench.sample_parity(w, A_np, p_np, r_np, w.M, (q_o, s_o), qg, sg)
    assert ok["pass"] and ok["checked"] == "q and s, every element"
    part = bench.sample_parity(w, A_np, p_np, r_np, 10, oracle.dualmv(A_np[:10], p_np,
                                                                        r_np[:10], N=w.N),
                               qg, sg)
    assert part["pass"] and part["checked"] == "q of the first 10 rows"
    bad = sg.copy()
    bad[5] = bad[5] + (7 if dtype == "i32" else 1.0)
    assert not bench.sample_parity(w, A_np, p_np, r_np, w.M, (q_o, s_o), qg, bad)["pass"]
