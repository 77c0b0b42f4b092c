#!/usr/bin/env python3
"""Benchmark of the fused dual matrix-vector product (BICG: q = A p, s = A^T r).

One step = one dualmv call over the whole workload (default: the 16384 x
16384 fp32 matrix, 1 GiB, seeded uniform[-1, 1)).  Prints ONE JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   (the CPU oracle, timed on the host)

Metric: effective bandwidth = (bytes of the logical A, of p and r read and of
q and s written) / device time, in GB/s (1e9 B/s).  The default inputs (1 GiB)
are larger than L2 (129 MB), so consecutive steps cannot hit in L2.  A
workload that fits in twice the L2 is timed call by call instead, with a
256 MiB buffer written between calls (outside the events) to evict it, and a
hot-L2 figure is added from a CUDA graph of 100 back-to-back calls.  Device
time comes from CUDA events on the launching stream, bracketed by a barrier
and a device synchronisation; with several ranks the slowest rank's time
counts.
Per-step times are also summarised with the trimmed mean of Eq. 3
(R timings sorted, k lowest and k highest dropped).

Multi-GPU: each rank runs its own copy of the workload on its own GPU (the
problems are independent; no data-path collective) and ``value`` counts the
bytes of all ranks: weak scaling.
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
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "dualmv effective HBM GB/s (bytes of A+vectors / device time) and % of GB300 peak"
DEFAULT_WORKLOAD = "f32_16384x16384"
FALLBACK_HBM_GBS = 6800.0
_CSRC = "paper_2512_22147_gb300/csrc/"
# Device sources of each streaming-kernel family: a traffic record stays
# valid while these are unchanged and the live call launches the same shape.
KERNEL_FAMILIES = {
    "dualmv_stream_kernel": (_CSRC + "dualmv_kernels.cuh",),
    "dualmv_stream_f64e_kernel": (_CSRC + "dualmv_kernels.cuh", _CSRC + "dualmv_f64e.cuh"),
    "dualmv_wide_i32_kernel": (_CSRC + "dualmv_kernels.cuh", _CSRC + "dualmv_wide.cuh"),
    "dualmv_small_cluster_kernel": (_CSRC + "dualmv_kernels.cuh", _CSRC + "dualmv_atax.cuh",
                                    _CSRC + "dualmv_small.cuh"),
}
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
FLUSH_BYTES = 256 << 20      # written between timed calls of an L2-sized workload
GRAPH_CALLS = 100            # calls captured in one CUDA graph (hot-L2 figure)
GB300_L2_BYTES = 126 << 20   # L2 size used when no GPU can be asked (reference arm on a CPU)


# ------------------------------------------------------------- helpers ----

def trimmed_mean(times, k: int) -> float:
    """Eq. 3: sort the R timings, drop the k lowest and k highest, average."""
    t = sorted(times)
    if k < 0 or len(t) <= 2 * k:
        raise ValueError("trimmed mean needs R > 2k")
    mid = t[k:len(t) - k]
    return sum(mid) / len(mid)


def kernel_family(name: str) -> str:
    """'dualmv_stream_f64e_kernel' from 'dmv::dualmv_stream_f64e_kernel<8, ...>'."""
    base = name.split("<")[0]
    return base.split("::")[-1]


def kernel_shape(name: str):
    """(warps, rows per warp, stages) from an ncu kernel name, by family."""
    args = [a.strip() for a in name.split("<", 1)[1].rstrip(">").split(",")]
    fam = kernel_family(name)
    if fam == "dualmv_stream_kernel":   # <T, W, RPW, STAGES, ...>
        return tuple(int(a) for a in args[1:4])
    if fam == "dualmv_small_cluster_kernel":   # <VPL, D>
        return tuple(int(a) for a in args[0:2])
    return tuple(int(a) for a in args[0:3])   # f64e and wide: <W, RPW, STAGES, ...>


def kernel_source_hash(family: str) -> str:
    h = hashlib.sha256()
    for rel in KERNEL_FAMILIES[family]:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def measured_peak():
    """(GB/s, source) from the generated MEASURED_PEAKS.json, else the
    fallback figure."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def recorded_traffic(workload: str, family: str | None = None, shape=None):
    """DRAM bytes per launch of the streaming kernel from a committed ncu
    capture, if it was taken on the current source of the kernel family the
    live call launched, with the same shape; else None."""
    try:
        with open(TRAFFIC_FILE) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    ent = rec.get(workload)
    if not ent or "kernel" not in ent:
        return None
    fam = kernel_family(ent["kernel"])
    if fam not in KERNEL_FAMILIES or ent.get("kernel_source_hash") != kernel_source_hash(fam):
        return None
    if family is not None and (fam != family or (
            shape is not None and kernel_shape(ent["kernel"]) != tuple(shape))):
        return None
    return ent.get("dram_bytes_per_launch")


_UNIT_SCALE = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12,
               "B": 1.0, "KB": 1e3, "MB": 1e6, "GB": 1e9,
               "nsecond": 1e-3, "usecond": 1.0, "msecond": 1e3, "second": 1e6,
               "ns": 1e-3, "us": 1.0, "ms": 1e3, "s": 1e6}


def parse_launch_list(path: str):
    """Launches of an ncu ``--csv --log-file`` metrics capture:
    ``[(id, kernel name, {metric: value in bytes or microseconds})]`` in
    launch order."""
    import csv
    with open(path, newline="") as f:
        lines = [ln for ln in f if ln.startswith('"')]
    rows = list(csv.reader(lines))
    hdr = rows[0]
    ix = {h: i for i, h in enumerate(hdr)}
    launches = {}
    for row in rows[1:]:
        lid = int(row[ix["ID"]])
        name = row[ix["Kernel Name"]]
        unit = row[ix["Metric Unit"]]
        val = float(row[ix["Metric Value"]].replace(",", ""))
        ent = launches.setdefault(lid, (name, {}))
        ent[1][row[ix["Metric Name"]]] = val * _UNIT_SCALE.get(unit, 1.0)
    return [(lid, n, m) for lid, (n, m) in sorted(launches.items())]


def short_kernel_name(name: str) -> str:
    name = name.split("(")[0]
    return name[5:] if name.startswith("void ") else name


def launch_table(launches):
    """Per kernel of a parsed launch list: [launches, total us, DRAM bytes]."""
    per = {}
    for _, name, m in launches:
        k = short_kernel_name(name)
        e = per.setdefault(k, [0, 0.0, 0.0])
        e[0] += 1
        e[1] += m.get("gpu__time_duration.sum", 0.0)
        e[2] += m.get("dram__bytes_read.sum", 0.0) + m.get("dram__bytes_write.sum", 0.0)
    return per


def summarize_launches(csv_path: str, command: str) -> str:
    """Markdown summary of an ncu launch list taken with
    ``--metrics gpu__time_duration.sum`` alone (one pass per launch, so it is
    safe on the full workload): per kernel its launches, total time and
    share.  ncu serialises launches and runs them cold: compare shares."""
    per = launch_table(parse_launch_list(csv_path))
    total = sum(e[1] for e in per.values()) or 1.0
    out = [f"Command (from the repository root, on one GB300; the plain command exited 0 "
           f"first):\n\n```\n{command}\n```\n",
           "| kernel | launches | total us | share | us / launch |",
           "|---|---|---|---|---|"]
    for k, (cnt, us, _) in sorted(per.items(), key=lambda kv: -kv[1][1]):
        out.append(f"| `{k[:120]}` | {cnt} | {us:.1f} | {100 * us / total:.1f} % | "
                   f"{us / cnt:.2f} |")
    return "\n".join(out)


def record_traffic(csv_path: str, workload: str, command: str, full_bytes: int,
                   case_bytes: int, case: str) -> str:
    """From a capture of the streaming kernel alone on a small case of
    ``workload`` (ncu ``-k`` one kernel, ``-c`` a few launches, DRAM and L2
    counters): its DRAM bytes (read + write) per launch, scaled to a full
    launch by the algorithmic bytes (``full_bytes / case_bytes``; A's bytes
    dominate and its traffic grows in proportion), written into the traffic
    record with the current kernel-source hash.  Returns a markdown summary
    of the captured counters."""
    launches = parse_launch_list(csv_path)
    per = launch_table(launches)
    stream = [k for k in per if kernel_family(k).startswith(("dualmv_stream", "dualmv_wide",
                                                             "dualmv_small_cluster"))]
    if len(stream) != 1:
        raise ValueError(f"expected one streaming kernel in the capture, found {stream}")
    n, us, dram = per[stream[0]]
    scale = full_bytes / case_bytes
    rec = {}
    if os.path.exists(TRAFFIC_FILE):
        with open(TRAFFIC_FILE) as f:
            rec = json.load(f)
    rec[workload] = {
        "kernel_source_hash": kernel_source_hash(kernel_family(stream[0])),
        "kernel": stream[0],
        "dram_bytes_per_launch": int(round(dram / n * scale)),
        "how": (f"ncu capture of the streaming kernel alone (-k, {n} launch(es)) on {case}: "
                f"dram__bytes_read.sum + dram__bytes_write.sum per launch = "
                f"{dram / n:.0f} B for {case_bytes} algorithmic bytes, scaled by "
                f"{scale:.4f} to the full workload's {full_bytes} algorithmic bytes"),
    }
    with open(TRAFFIC_FILE, "w") as f:
        json.dump(rec, f, indent=1)
        f.write("\n")
    metrics = {}
    for _, name, m in launches:
        if short_kernel_name(name) == stream[0]:
            for key, val in m.items():
                metrics.setdefault(key, []).append(val)
    out = [f"Command (from the repository root, on one GB300; the plain command exited 0 "
           f"first):\n\n```\n{command}\n```\n",
           f"Kernel `{stream[0]}`, {n} launch(es) on {case} ({case_bytes} algorithmic bytes).\n",
           "| metric | per launch |", "|---|---|"]
    for key in sorted(metrics):
        out.append(f"| {key} | {sum(metrics[key]) / len(metrics[key]):.6g} |")
    out.append(f"\nDRAM read + write per launch: {dram / n / case_bytes:.4f} x the algorithmic "
               f"bytes; scaled to the full workload: {int(round(dram / n * scale))} B.")
    return "\n".join(out)


class ClockSampler:
    """nvidia-smi clock and throttle-reason samples while the timed region runs."""

    QUERY = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def start(self):
        import tempfile
        fd, self.path = tempfile.mkstemp(prefix="dualmv_clocks_", suffix=".csv")
        os.close(fd)
        cmd = ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
               "-lms", "100"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"),
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"],
                    "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 10:
                    rows.append(parts)
        os.unlink(self.path)
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[6:10]) if v == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def gpu_uuid(torch, dev):
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:  # noqa: BLE001 - older torch: sample the default GPU
        return None


def workload_from_args(inputs, args):
    """The named workload, optionally resized (for small profiling cases)."""
    w = inputs.WORKLOADS.get(args.workload) or inputs.OP_WORKLOADS[args.workload]
    kw = {}
    for k in ("M", "N", "lda", "batch"):
        v = getattr(args, k)
        if v is not None:
            kw[k] = v
    if "N" in kw and "lda" not in kw:
        kw["lda"] = kw["N"]
    if kw:
        w = w.scaled(name=w.name + "_resized_" + "_".join(f"{k}{v}" for k, v in kw.items()),
                     **kw)
    return w


# ---------------------------------------------------------- distributed ---

def dist_setup(torch, backend):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
    return world, rank, local


def max_over_ranks(torch, value: float, world: int, device) -> float:
    if world == 1:
        return value
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# --------------------------------------------------------------- native ---

def make_call(torch, dm, inputs, w, dev):
    """The closure that runs one step of workload ``w`` and the tensors it
    uses: ``(call, state)``; state holds A, p, r, q, s for the dual product."""
    if w.op == "bicg":
        A, p, r = inputs.generate(w, dev)
        Av = A[..., : w.N]
        q, s = inputs.empty_outputs(w, dev)

        def call():
            dm.dualmv(Av, p, r, q=q, s=s)
        return call, {"A": A, "p": p, "r": r, "q": q, "s": s}
    if w.op == "gesummv":
        A, Bm, x = inputs.generate_gesummv(w, dev)
        y = torch.empty(w.M, dtype=A.dtype, device=dev)

        def call():
            dm.gesummv(A[:, : w.N], Bm[:, : w.N], x, alpha=1.5, beta=1.2, y=y)
        return call, {"A": A, "B": Bm, "x": x, "y": y}
    if w.op == "atax":
        A, x = inputs.generate_atax(w, dev)
        y = torch.empty(w.N, dtype=A.dtype, device=dev)

        def call():
            dm.atax(A[:, : w.N], x, y=y)
        return call, {"A": A, "x": x, "y": y}
    # gemver: x and w accumulate in place from call to call
    A, u1, v1, u2, v2, wv, x, y, z = inputs.generate_gemver(w, dev)

    def call():
        dm.gemver(A[:, : w.N], u1, v1, u2, v2, wv, x, y, z, alpha=1.5, beta=1.2,
                  update_A=w.update_a)
    return call, {"A": A, "x": x, "w": wv}


def timed_region(torch, call, K, W, flush, stream, dev, world, uuid):
    """The contract's timed region.  The clock sampler starts, then the W
    warm-up calls run right before the region (so the GPU is at speed when
    it opens, not idle after the sampler's start-up pause); a barrier and a
    device synchronisation on both sides; K calls back to back between two
    events, or, with ``flush`` (an L2-sized workload), each call between its
    own events after an L2-evicting write outside them.  Returns (region
    milliseconds, clock record)."""
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.3)  # let the sampler start before the GPU work
    for _ in range(W):
        call()
    torch.cuda.synchronize(dev)
    barrier(world)
    torch.cuda.synchronize(dev)
    if flush is None:
        ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        ev[0].record(stream)
        for _ in range(K):
            call()
        ev[1].record(stream)
    else:
        flushed = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(K)]
        for ev0, ev1 in flushed:
            flush.zero_()
            ev0.record(stream)
            call()
            ev1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clocks = sampler.stop()
    if flush is None:
        return ev[0].elapsed_time(ev[1]), clocks
    return sum(a.elapsed_time(b) for a, b in flushed), clocks


def instrumented_calls(torch, dm, call, n, flush, stream, dev, per_kernel: bool):
    """``n`` more calls, each between its own events; with ``per_kernel`` the
    library also records events around its streaming kernel on the stream it
    runs on (dualmv_record_kernel_events).  Returns (per-call ms, kernel ms);
    without ``per_kernel`` the kernel times are the whole calls."""
    call_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(n)]
    kern_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(n)]
    # torch creates a CUDA event lazily on its first record; the library
    # records the kernel events itself, so make them exist first.
    for ks, ke in kern_ev:
        ks.record(stream)
        ke.record(stream)
    torch.cuda.synchronize(dev)
    for i in range(n):
        ks, ke = kern_ev[i]
        if flush is not None:
            flush.zero_()
        if per_kernel:
            dm.dualmv_record_kernel_events(ks.cuda_event, ke.cuda_event)
        else:
            ks.record(stream)
        call_ev[i][0].record(stream)
        call()
        call_ev[i][1].record(stream)
        if not per_kernel:
            ke.record(stream)
    torch.cuda.synchronize(dev)
    return ([a.elapsed_time(b) for a, b in call_ev], [a.elapsed_time(b) for a, b in kern_ev])


def streaming_kernel_name(dm, w):
    """(name, family, shape) of the streaming kernel the last dual product
    launched, for the roofline record."""
    kernel_name = f"whole {w.op} call"
    family, shape = None, None
    if w.op != "bicg":
        return kernel_name, family, shape
    kernel_name = "dualmv_stream_kernel"
    vi = dm.dualmv_last_variant()
    if vi >= 0:
        v = dm.dualmv_variant_info({"f32": 0, "f64": 1, "i32": 2}[w.dtype], vi)
        family = {dm.DUALMV_KERNEL_STREAM: "dualmv_stream_kernel",
                  dm.DUALMV_KERNEL_F64E: "dualmv_stream_f64e_kernel",
                  dm.DUALMV_KERNEL_WIDE: "dualmv_wide_i32_kernel"}[v.kernel]
        shape = (v.warps, v.rows_per_warp, v.stages)
        kernel_name = family + f"<warps {v.warps}, rows {v.rows_per_warp}, stages {v.stages}>"
    else:  # batched (the default kernel), unaligned rows, or plain loads
        kind = dm.dualmv_last_kernel()
        kernel_name = {
            dm.DUALMV_KERNEL_PHASED: ("dualmv_stream_f64e_phased_kernel" if w.dtype == "f64"
                                      else "dualmv_stream_phased_kernel"),
            dm.DUALMV_KERNEL_PLAIN: "dualmv_stream_kernel (plain loads)",
            dm.DUALMV_KERNEL_CLUSTER: "dualmv_small_cluster_kernel (one cluster of 16 CTAs)",
        }.get(kind, kernel_name)
        if w.batched and kind in (dm.DUALMV_KERNEL_STREAM, dm.DUALMV_KERNEL_F64E):
            family = {dm.DUALMV_KERNEL_STREAM: "dualmv_stream_kernel",
                      dm.DUALMV_KERNEL_F64E: "dualmv_stream_f64e_kernel"}[kind]
        if kind == dm.DUALMV_KERNEL_CLUSTER:
            family = "dualmv_small_cluster_kernel"
    return kernel_name, family, shape


def launches_per_call(torch, dm, inputs, w, dev) -> int:
    """Kernels of this library one call launches."""
    plan = dm.dualmv_plan(w.M, w.N, w.nbatch, inputs.ELEM_BYTES[w.dtype],
                          inputs.OUT_BYTES[w.dtype],
                          torch.cuda.get_device_properties(dev).multi_processor_count)
    n = 1 + (1 if (plan.bands > 1 or plan.grid > 1) else 0)
    if w.op == "bicg" and dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_CLUSTER:
        n = 1   # one cluster computes both outputs, no combine kernel
    if w.op == "gesummv":   # two row passes, then one kernel adds their partials into y
        return 3
    if w.op == "atax":      # a row pass and a column pass
        return 2 * n
    if w.op == "gemver":    # u.y dots, column pass, x update, row pass, w update
        return 5
    return n


def read_ceiling(torch, dm, dev, stream, reps=10, nbytes=2 << 30):
    """Read-only bandwidth of this GPU: the library's read probe (16-byte
    loads over every SM) on a 2 GiB buffer, larger than L2, timed with
    events on the launching stream after three warm-up passes."""
    buf = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    out = torch.zeros(1, dtype=torch.int32, device=dev)
    sp = stream.cuda_stream

    def one():
        rc = dm.dualmv_read_probe(buf.data_ptr(), nbytes, out.data_ptr(), sp)
        if rc != dm.DUALMV_SUCCESS:
            raise RuntimeError(f"dualmv_read_probe: status {rc}")
    for _ in range(3):
        one()
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        one()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    gbs = nbytes * reps / (e0.elapsed_time(e1) * 1e-3) / 1e9
    del buf, out
    return {"gbs": round(gbs, 1), "bytes": nbytes, "reps": reps,
            "how": "dualmv_read_probe: 16-byte loads, 8 in flight per thread, 2048 threads per "
                   "SM, over a 2 GiB buffer; CUDA events on the launching stream"}


def run_native(args):
    import torch

    world, rank, local = dist_setup(torch, "nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import paper_2512_22147_gb300 as dm
    from paper_2512_22147_gb300 import inputs

    w = workload_from_args(inputs, args)
    stream = torch.cuda.current_stream(dev)
    nbytes = w.bytes_counted()
    call, st = make_call(torch, dm, inputs, w, dev)

    if args.variant is not None:   # force one compiled kernel variant (profiling)
        dm.dualmv_set_variant({"f32": 0, "f64": 1, "i32": 2}[w.dtype], args.variant)
    tuned = None
    if args.tune:
        if w.op != "bicg":
            raise SystemExit("--tune applies to the dual product (one problem or a batch)")
        t0 = time.time()
        Av = st["A"][..., : w.N]
        rep = dm.tune(Av, st["p"], st["r"], repeats=30, trim=3, max_rounds=4, candidates=8,
                      min_gain=0.01, flush_l2=flush_needed(torch, nbytes, dev))
        torch.cuda.synchronize(dev)
        v = dm.dualmv_variant_info({"f32": 0, "f64": 1, "i32": 2}[w.dtype], rep["best"])
        tuned = {k: (float(f"{val:.6g}") if isinstance(val, float) else val)
                 for k, val in rep.items() if k not in ("q", "s", "trace")}
        tuned["trace"] = [{k: (float(f"{val:.6g}") if isinstance(val, float) else val)
                           for k, val in stp.items()} for stp in rep["trace"]]
        tuned["variant"] = {f: getattr(v, f) for f, _ in v._fields_}
        tuned["seconds"] = round(time.time() - t0, 2)

    K = args.steps
    flush = None
    if flush_needed(torch, nbytes, dev):   # the operands could stay in L2 between calls
        flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    uuid = gpu_uuid(torch, dev)

    region_ms, clocks = timed_region(torch, call, K, args.warmup, flush, stream, dev, world,
                                     uuid)
    if dm.device_fault() != dm.DUALMV_SUCCESS:
        raise RuntimeError("device fault during the timed region")
    region_ms = max_over_ranks(torch, region_ms, world, dev)
    ms_per_step = region_ms / K
    value = world * nbytes * K / (region_ms * 1e-3) / 1e9

    # Instrumented region: per-call events for the trimmed mean of Eq. 3 and
    # the streaming kernel's own time for the roofline.
    Ki = min(K, args.instrumented_steps)
    step_ms, kern_ms = instrumented_calls(torch, dm, call, Ki, flush, stream, dev,
                                          per_kernel=w.op == "bicg")
    if dm.device_fault() != dm.DUALMV_SUCCESS:
        raise RuntimeError("device fault during the instrumented region")
    peak, peak_src = measured_peak()
    kern_avg_ms = sum(kern_ms) / len(kern_ms)
    kernel_name, family, shape = streaming_kernel_name(dm, w)
    achieved = nbytes / (kern_avg_ms * 1e-3) / 1e9
    traffic = recorded_traffic(args.workload, family, shape) if family else None
    ceiling = None if args.no_read_ceiling else read_ceiling(torch, dm, dev, stream)

    hot = hot_l2_graph(torch, call, nbytes, dev) if flush is not None else None

    # End to end through the same public call with host buffers: pinned host
    # inputs copied in, the call, results copied out, every step.
    e2e = None
    if not args.no_e2e and w.op == "bicg":
        e2e = run_e2e(torch, dm, w, st["A"], st["p"], st["r"], dev, stream, args.e2e_steps,
                      uuid)

    deterministic = bitwise_repeat(torch, call, st, w, dev)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and w.op == "bicg":
        cpu = cpu_baseline(w, st["A"], st["p"], st["r"], args.cpu_seconds, st["q"], st["s"],
                           parallel_s=args.cpu_parallel_seconds)

    configs = None
    if (world == 1 and not args.no_configs and w.op == "bicg" and args.variant is None
            and not args.tune and w.name in inputs.WORKLOADS):
        del st, call
        torch.cuda.empty_cache()
        configs = {}
        for name, wc in inputs.WORKLOADS.items():
            if name == w.name:
                continue
            configs[name] = measure_config(torch, dm, inputs, wc, dev, stream, args.warmup,
                                           uuid, peak, ceiling, args.config_seconds)
            torch.cuda.empty_cache()

    out = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": w.dtype,
        "data": "synthetic",
        "config": workload_config(w, nbytes, flush is not None, world, args.variant),
        "pct_of_peak": round(100.0 * value / (world * peak), 2),
        "trimmed_mean_ms": round(trimmed_mean(step_ms, 3) if Ki > 6 else statistics.mean(step_ms), 5),
        "median_step_ms": round(statistics.median(step_ms), 5),
        "min_step_ms": round(min(step_ms), 5),
        "roofline": {
            "bound": "hbm",
            "kernel": kernel_name,
            "achieved": round(achieved, 2),
            "peak": peak,
            "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
            else "fallback 6.8 TB/s",
            "unit": "GB/s",
            "frac": round(achieved / peak, 4),
            "traffic": traffic,
            "algorithmic_bytes_per_launch": nbytes,
            "kernel_avg_ms": round(kern_avg_ms, 5),
            **({"read_ceiling": ceiling,
                "frac_of_read_ceiling": round(achieved / ceiling["gbs"], 4)} if ceiling else {}),
        },
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches_per_call(torch, dm, inputs, w, dev) * K,
        "deterministic": deterministic,
        "instrumented_steps": Ki,
        "clocks": clocks,
    }
    if hot is not None:
        out["hot_l2_graph"] = hot
    if tuned is not None:
        out["tuned"] = tuned
    if configs is not None:
        out["configs"] = configs
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def bitwise_repeat(torch, call, st, w, dev):
    """Two more calls compared bit for bit (None for GEMVER, whose x and w
    change from call to call)."""
    if w.op == "bicg":
        call()
        q1, s1 = st["q"].clone(), st["s"].clone()
        call()
        torch.cuda.synchronize(dev)
        return bool(torch.equal(q1, st["q"]) and torch.equal(s1, st["s"]))
    if w.op in ("gesummv", "atax"):
        call()
        y1 = st["y"].clone()
        call()
        torch.cuda.synchronize(dev)
        return bool(torch.equal(y1, st["y"]))
    return None


def measure_config(torch, dm, inputs, w, dev, stream, W, uuid, peak, ceiling, target_s):
    """One more of the benchmark's dual-product workloads, measured in the
    same process as the headline: W warm-up calls, then K calls timed as the
    headline is (K sized for about ``target_s`` seconds of GPU time), the
    streaming kernel timed on its own stream over 30 further calls, the
    clocks sampled during the timed region, the outputs compared with the
    oracle (every element; the first 8 problems of a batch) and two further
    calls compared bit for bit."""
    nbytes = w.bytes_counted()
    call, st = make_call(torch, dm, inputs, w, dev)
    flush = None
    if flush_needed(torch, nbytes, dev):
        flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    for _ in range(max(W, 3)):   # size K from the warm-up calls' time
        call()
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(5):
        call()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    est_ms = max(e0.elapsed_time(e1) / 5, 1e-3)
    K = int(min(3000, max(20, math.ceil(target_s * 1e3 / est_ms))))
    region_ms, clocks = timed_region(torch, call, K, W, flush, stream, dev, 1, uuid)
    step_ms, kern_ms = instrumented_calls(torch, dm, call, 30, flush, stream, dev, True)
    kernel_name, _, _ = streaming_kernel_name(dm, w)
    fault = dm.device_fault()
    value = nbytes * K / (region_ms * 1e-3) / 1e9
    kern_avg_ms = sum(kern_ms) / len(kern_ms)
    achieved = nbytes / (kern_avg_ms * 1e-3) / 1e9
    hot = hot_l2_graph(torch, call, nbytes, dev) if flush is not None else None
    deterministic = bitwise_repeat(torch, call, st, w, dev)
    n = min(w.batch, 8) if w.batched else w.M
    A_np = st["A"][:n].cpu().numpy() if w.batched else st["A"].cpu().numpy()
    p_np = st["p"][:n].cpu().numpy() if w.batched else st["p"].cpu().numpy()
    r_np = st["r"][:n].cpu().numpy() if w.batched else st["r"].cpu().numpy()
    import oracle
    outs = (oracle.dualmv_batched(A_np, p_np, r_np, N=w.N) if w.batched
            else oracle.dualmv(A_np, p_np, r_np, N=w.N))
    parity = sample_parity(w, A_np, p_np, r_np, n, outs, st["q"].cpu().numpy(),
                           st["s"].cpu().numpy())
    out = {
        "value": round(value, 2), "unit": "GB/s",
        "pct_of_peak": round(100.0 * value / peak, 2),
        "ms_per_step": round(region_ms / K, 5), "steps": K, "warmup": W,
        "bytes_per_step": nbytes,
        "config": {"M": w.M, "N": w.N, "lda": w.lda, "batch": w.batch, "dtype": w.dtype,
                   "distribution": w.dist, "seed": w.seed},
        "l2": ("inputs larger than L2 (no flush needed)" if flush is None else
               f"L2 flushed: {FLUSH_BYTES >> 20} MiB written before each call, outside its "
               "events"),
        "trimmed_mean_ms": round(trimmed_mean(step_ms, 3), 5),
        "median_step_ms": round(statistics.median(step_ms), 5),
        "min_step_ms": round(min(step_ms), 5),
        "kernel": kernel_name,
        "kernel_avg_ms": round(kern_avg_ms, 5),
        "kernel_frac": round(achieved / peak, 4),
        **({"kernel_frac_of_read_ceiling": round(achieved / ceiling["gbs"], 4)} if ceiling
           else {}),
        "gpu_launches": launches_per_call(torch, dm, inputs, w, dev) * K,
        "parity": parity,
        "deterministic": deterministic,
        "device_fault": fault != dm.DUALMV_SUCCESS,
        "clocks": clocks,
    }
    if hot is not None:
        out["hot_l2_graph"] = hot
    del st, call, flush
    return out


def workload_config(w, nbytes: int, flushed: bool, world: int, variant=None) -> dict:
    """The JSON line's ``config``: the workload and how it is timed.  Both
    arms print the same dict for the same workload."""
    return {
        "workload": w.name, "op": w.op, "M": w.M, "N": w.N, "lda": w.lda,
        "batch": w.batch, "dtype": w.dtype, "distribution": w.dist, "seed": w.seed,
        "bytes_per_step": nbytes,
        "l2": (f"L2 flushed: {FLUSH_BYTES >> 20} MiB written before each call, "
               "outside its events" if flushed else
               "inputs larger than L2 (no flush needed)"),
        "parallelism": f"replicas x{world}",
        **({"variant": variant} if variant is not None else {}),
    }


def flush_needed(torch, nbytes: int, dev) -> bool:
    """True when a workload's operands could stay in L2 between calls."""
    return nbytes <= 2 * torch.cuda.get_device_properties(dev).L2_cache_size


def hot_l2_graph(torch, call, nbytes, dev, reps=20):
    """Per-call time of GRAPH_CALLS back-to-back calls captured in one CUDA
    graph and replayed ``reps`` times: the operands stay in L2 and the host
    launch cost is gone, which leaves the kernels' own latency."""
    try:
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))
        with torch.cuda.stream(side):
            call()
        torch.cuda.current_stream(dev).wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(GRAPH_CALLS):
                call()
        g.replay()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize(dev)
    except Exception as ex:  # capture is a measurement extra; report why it failed
        return {"error": f"{type(ex).__name__}: {ex}"[:300]}
    per_call_ms = e0.elapsed_time(e1) / (reps * GRAPH_CALLS)
    return {"calls_per_graph": GRAPH_CALLS, "replays": reps,
            "per_call_us": round(per_call_ms * 1e3, 3),
            "GBs": round(nbytes / (per_call_ms * 1e-3) / 1e9, 2)}


def run_e2e(torch, dm, w, A, p, r, dev, stream, steps, uuid=None):
    Ah = A.cpu().pin_memory()
    ph = p.cpu().pin_memory()
    rh = r.cpu().pin_memory()
    Ad = torch.empty_like(A)
    pd = torch.empty_like(p)
    rd = torch.empty_like(r)
    q, s = dm.dualmv(Ad[..., : w.N].copy_(A[..., : w.N]), pd.copy_(p), rd.copy_(r))
    qh = torch.empty(q.shape, dtype=q.dtype).pin_memory()
    sh = torch.empty(s.shape, dtype=s.dtype).pin_memory()
    torch.cuda.synchronize(dev)
    start = torch.cuda.Event(enable_timing=True)
    stop = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        Ad.copy_(Ah, non_blocking=True)
        pd.copy_(ph, non_blocking=True)
        rd.copy_(rh, non_blocking=True)
        dm.dualmv(Ad[..., : w.N], pd, rd, q=q, s=s)
        qh.copy_(q, non_blocking=True)
        sh.copy_(s, non_blocking=True)
    stop.record(stream)
    torch.cuda.synchronize(dev)
    ms = start.elapsed_time(stop) / steps
    h2d = Ah.numel() * Ah.element_size() + ph.numel() * ph.element_size() \
        + rh.numel() * rh.element_size()
    d2h = qh.numel() * qh.element_size() + sh.numel() * sh.element_size()
    return {"value": round(w.bytes_counted() / (ms * 1e-3) / 1e9, 2), "unit": "GB/s",
            "ms_per_step": round(ms, 4), "steps": steps,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "how": "pinned host A, p, r copied to the GPU, dualmv through the C ABI, q and s "
                   "copied back, all on one stream inside CUDA events",
            "host_placement": host_placement(Ah.data_ptr(), h2d, uuid)}


def _cpulist(text: str) -> set:
    cpus = set()
    for part in text.strip().split(","):
        if part:
            a, _, b = part.partition("-")
            cpus |= set(range(int(a), int(b or a) + 1))
    return cpus


def host_placement(ptr: int, nbytes: int, uuid=None, samples: int = 64):
    """Where the pinned input buffer lives: the NUMA nodes of a sample of its
    pages (move_pages with no target node reports each page's node), the
    nodes of the CPUs this process may run on, and the NUMA node sysfs gives
    for the GPU's PCI function.  Linux only; fields it cannot read are null."""
    import ctypes
    import platform
    out = {"buffer_page_nodes": None, "process_cpu_nodes": None, "gpu_numa_node": None}
    try:
        nr = {"aarch64": 239, "x86_64": 279}[platform.machine()]
        libc = ctypes.CDLL(None, use_errno=True)
        ps = os.sysconf("SC_PAGE_SIZE")
        addrs = [(ptr + k * (nbytes // samples)) & ~(ps - 1) for k in range(samples)]
        arr = (ctypes.c_void_p * samples)(*addrs)
        status = (ctypes.c_int * samples)()
        if libc.syscall(nr, 0, ctypes.c_ulong(samples), arr, None, status, 0) == 0:
            counts = {}
            for v in status:
                counts[str(v)] = counts.get(str(v), 0) + 1
            out["buffer_page_nodes"] = counts
    except (KeyError, OSError, AttributeError):
        pass
    try:
        allowed = os.sched_getaffinity(0)
        nodes = []
        base = "/sys/devices/system/node"
        for n in sorted(os.listdir(base)):
            if n.startswith("node"):
                with open(os.path.join(base, n, "cpulist")) as f:
                    if _cpulist(f.read()) & allowed:
                        nodes.append(int(n[4:]))
        out["process_cpu_nodes"] = nodes
    except OSError:
        pass
    try:
        cmd = ["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader"]
        if uuid:
            cmd += ["-i", uuid]
        bus = subprocess.run(cmd, capture_output=True, text=True,
                             timeout=20).stdout.strip().splitlines()[0]
        dom, rest = bus.split(":", 1)
        with open(f"/sys/bus/pci/devices/{(dom[-4:] + ':' + rest).lower()}/numa_node") as f:
            out["gpu_numa_node"] = int(f.read().strip())
    except (OSError, ValueError, IndexError, subprocess.SubprocessError):
        pass
    return out


# ------------------------------------------------------- CPU (oracle) ----

def oracle_sample(w, A_np, p_np, r_np, budget_s: float):
    """Times the oracle on leading rows of the workload (of each problem,
    batched: leading problems), growing the sample until it takes about
    ``budget_s`` seconds or covers the whole workload; a whole workload that
    takes less than the budget is timed over repeated passes.  Returns
    (bytes per second, seconds, description, n, oracle outputs)."""
    import oracle
    from paper_2512_22147_gb300 import inputs

    e, o = inputs.ELEM_BYTES[w.dtype], inputs.OUT_BYTES[w.dtype]
    units = w.batch if w.batched else w.M

    def run(n):
        if w.batched:
            outs = oracle.dualmv_batched(A_np[:n], p_np[:n], r_np[:n], N=w.N)
            return outs, n * (w.M * w.N * e + (w.M + w.N) * (e + o))
        outs = oracle.dualmv(A_np[:n], p_np, r_np[:n], N=w.N)
        return outs, n * w.N * e + (n + w.N) * (e + o)

    n = max(1, min(units, 64))
    while True:
        t0 = time.perf_counter()
        outs, nbytes = run(n)
        dt = time.perf_counter() - t0
        if dt >= budget_s or n >= units:
            break
        grow = max(2.0, min(8.0, budget_s / max(dt, 1e-3)))
        n = min(units, int(math.ceil(n * grow)))
    passes = 1
    if dt < 0.5 * budget_s:
        passes = max(1, min(10000, int(budget_s / max(dt, 1e-6))))
        t0 = time.perf_counter()
        for _ in range(passes):
            outs, nbytes = run(n)
        dt = time.perf_counter() - t0
        nbytes *= passes
    what = (f"first {n} of {units} {'problems' if w.batched else 'rows'} of {w.name}"
            f"{f', {passes} passes' if passes > 1 else ''}, "
            f"single-threaded C oracle (double/Dot2/int64 sums)")
    return nbytes / dt / 1e9, dt, what, n, outs


PARITY_TOL = {"f32": 1e-5, "f64": 1e-12, "i32": 0.0}


def sample_parity(w, A_np, p_np, r_np, n, outs, q_gpu, s_gpu):
    """Scaled error of the benchmark's own GPU outputs against the oracle's
    outputs on the sampled part: q of the sampled rows (problems), and s too
    when the sample is the whole workload.  Integer outputs must be equal."""
    import numpy as np
    import oracle

    q_o, s_o = outs
    whole = n >= (w.batch if w.batched else w.M)
    qg = q_gpu[:n]
    sg = s_gpu[:n] if w.batched else s_gpu
    if w.dtype == "i32":
        ok_q = np.array_equal(qg, q_o)
        ok_s = (not whole) or np.array_equal(sg, s_o)
        err = 0.0 if (ok_q and ok_s) else float("inf")
    else:
        def scaled(got, want, den):
            diff = np.abs(got.astype(np.float64) - want)
            z = den == 0
            if z.any() and (diff[z] != 0).any():
                return float("inf")
            return float((diff[~z] / den[~z]).max()) if (~z).any() else 0.0
        if w.batched:
            errs = []
            for b in range(n):
                qa, sa = oracle.absdot(A_np[b], p_np[b], r_np[b], N=w.N)
                errs += [scaled(qg[b], q_o[b], qa), scaled(sg[b], s_o[b], sa)]
            err = max(errs)
        else:
            qa, sa = oracle.absdot(A_np[:n], p_np, r_np[:n], N=w.N)
            err = scaled(qg, q_o, qa)
            if whole:
                err = max(err, scaled(sg, s_o, sa))
    checked = (f"q and s of the first {n} problems" if w.batched else
               ("q and s, every element" if whole else f"q of the first {n} rows"))
    return {"max_scaled_error": err, "tolerance": PARITY_TOL[w.dtype],
            "checked": checked, "pass": bool(err <= PARITY_TOL[w.dtype])}


def cpu_baseline(w, A, p, r, budget_s, q=None, s=None, parallel_s=0.0):
    A_np = A.cpu().numpy()
    p_np, r_np = p.cpu().numpy(), r.cpu().numpy()
    gbs, dt, what, n, outs = oracle_sample(w, A_np, p_np, r_np, budget_s)
    out = {"value": round(gbs, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
           "sample": what, "seconds": round(dt, 3), "host_cpus": os.cpu_count()}
    if q is not None:
        out["parity"] = sample_parity(w, A_np, p_np, r_np, n, outs, q.cpu().numpy(),
                                      s.cpu().numpy())
    if parallel_s > 0 and not w.batched:
        out["parallel"] = parallel_baseline(w, A_np, p_np, r_np, n, outs, parallel_s)
    return out


def parallel_baseline(w, A_np, p_np, r_np, n, outs, budget_s):
    """The oracle's loops on every host core (oracle/oracle_omp.c, OpenMP):
    the same rows as the single-core sample, repeated for about ``budget_s``
    seconds.  Each output is summed in the oracle's order, so the outputs
    must equal the oracle's bit for bit; that is checked too."""
    import numpy as np
    import oracle

    e, o = inputs_sizes(w)
    nbytes = n * w.N * e + (n + w.N) * (e + o)
    A_s, r_s = A_np[:n], r_np[:n]
    t0 = time.perf_counter()
    q_p, s_p = oracle.dualmv_omp(A_s, p_np, r_s, N=w.N)
    dt = time.perf_counter() - t0
    passes = max(1, min(1000, int(budget_s / max(dt, 1e-6))))
    t0 = time.perf_counter()
    for _ in range(passes):
        oracle.dualmv_omp(A_s, p_np, r_s, N=w.N)
    dt = time.perf_counter() - t0
    same = bool(np.array_equal(q_p, outs[0]) and np.array_equal(s_p, outs[1]))
    return {"value": round(nbytes * passes / dt / 1e9, 4), "unit": "GB/s",
            "cores": oracle.omp_threads(), "kind": "oracle loops on every host core (OpenMP)",
            "sample": f"first {n} of {w.M} rows of {w.name}, {passes} passes; A read twice "
                      "(rows for q, column blocks for s)",
            "seconds": round(dt, 3), "bitwise_equal_to_oracle": same}


def inputs_sizes(w):
    from paper_2512_22147_gb300 import inputs
    return inputs.ELEM_BYTES[w.dtype], inputs.OUT_BYTES[w.dtype]


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch

    from paper_2512_22147_gb300 import inputs
    w = workload_from_args(inputs, args)
    A, p, r = inputs.generate(w, "cpu")
    A_np, p_np, r_np = A.numpy(), p.numpy(), r.numpy()
    budget = args.cpu_seconds / max(1, args.steps + args.warmup)
    vals, secs = [], []
    what = ""
    for i in range(args.warmup + args.steps):
        gbs, dt, what, _, _ = oracle_sample(w, A_np, p_np, r_np, budget)
        if i >= args.warmup:
            vals.append(gbs)
            secs.append(dt)
    value = statistics.mean(vals)
    nbytes = w.bytes_counted()
    if torch.cuda.is_available():   # the native arm's rule for this GPU's L2
        flushed = flush_needed(torch, nbytes, 0)
    else:
        flushed = nbytes <= 2 * GB300_L2_BYTES
    del torch
    out = {
        "impl": "reference",
        "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * statistics.mean(secs), 4), "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": workload_config(w, nbytes, flushed, world, args.variant),
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": 1,
                         "kind": "oracle", "sample": what},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--instrumented-steps", type=int, default=300)
    ap.add_argument("--M", type=int, default=None, help="resize the workload (profiling)")
    ap.add_argument("--N", type=int, default=None)
    ap.add_argument("--lda", type=int, default=None)
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-parallel-seconds", type=float, default=3.0,
                    help="time budget of the all-core (OpenMP) oracle baseline; 0 skips it")
    ap.add_argument("--no-read-ceiling", action="store_true",
                    help="skip the read-only bandwidth probe")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other dual-product workloads (the 'configs' block)")
    ap.add_argument("--config-seconds", type=float, default=0.25,
                    help="GPU time of each other workload's timed region")
    ap.add_argument("--variant", type=int, default=None,
                    help="force this entry of the dtype's kernel-variant table")
    ap.add_argument("--tune", action="store_true",
                    help="run the variant tuner (Eq. 3-5) on the workload before warm-up; "
                         "the timed calls then use the variant it chose")
    ap.add_argument("--record-traffic", metavar="CSV", default=None,
                    help="from an ncu capture of the streaming kernel alone on the case that "
                         "--workload with --M/--N/--lda/--batch names, record its DRAM bytes "
                         "per launch scaled to the full --workload, then exit")
    ap.add_argument("--summarize-launches", metavar="CSV", default=None,
                    help="print a markdown summary of an ncu launch list (time only), then exit")
    ap.add_argument("--record-command", default="", help="the command that made the CSV")
    args = ap.parse_args(argv)
    if args.summarize_launches:
        print(summarize_launches(args.summarize_launches, args.record_command))
        return
    if args.record_traffic:
        from paper_2512_22147_gb300 import inputs
        case = workload_from_args(inputs, args)
        full = inputs.WORKLOADS.get(args.workload) or inputs.OP_WORKLOADS[args.workload]
        desc = (f"{case.M} x {case.N}, lda {case.lda}" + (f", batch {case.batch}" if case.batch
                                                           else "") + f", {case.dtype}")
        print(record_traffic(args.record_traffic, args.workload, args.record_command,
                             full.bytes_counted(), case.bytes_counted(), desc))
        return
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
