#!/usr/bin/env python
"""Benchmark of the exact integer GEMM C += A*B on one or more GB300s.

One "step" is one call of the public API on the whole workload: for the
default workload (int16 8192^3, the compute-bound roofline point) that is the
limb split of A and B plus the tcgen05 GEMM kernel.  Prints ONE JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gemmi|reference]
                    [--workload NAME] [--no-extra] [--cpu-seconds S]

--impl reference times the CPU oracle (the plain triple loop) on the host
cores, on bounded row samples of the same workload.  Under torchrun (N > 1)
every rank runs an independent replica of the workload (the GEMM has no
exchange step), rank 0 prints the aggregate.
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
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import gemm_inputs as gi  # noqa: E402

L2_BYTES = 129 * 2 ** 20
PROFILES = os.path.join(ROOT, "profiles")
# per kernel of the library: its CUDA symbol, the sources it is built from, and its bound
KERNEL_INFO = {
    "split": ("split_tma_kernel", ("split.cu", "ptx.cuh", "tc_common.cuh"), "hbm"),
    "tc_i16": ("tc_gemm_kernel<2>", ("gemm_tc.cu", "tc_common.cuh", "ptx.cuh"), "tensor"),
    "tc_i8": ("tc_gemm_kernel<1>", ("gemm_tc.cu", "tc_common.cuh", "ptx.cuh"), "tensor"),
    "skinny": ("skinny_kernel", ("skinny.cu", "ptx.cuh", "tc_common.cuh"), "hbm"),
    "fused_i16": ("fused_kernel", ("gemm_fused.cu", "tc_common.cuh", "ptx.cuh"), "hbm"),
    "srs": ("srs_add_kernel", ("requant.cu",), "hbm"),
    "tc_pair_i16": ("tc_pair_kernel<2>", ("gemm_pair.cu", "tc_common.cuh", "ptx.cuh", "ptx_pair.cuh"), "tensor"),
    "tc_pair_i8": ("tc_pair_kernel<1>", ("gemm_pair.cu", "tc_common.cuh", "ptx.cuh", "ptx_pair.cuh"), "tensor"),
    "tc_pair_i4": ("tc_pair_kernel<1,e4m3>", ("gemm_pair.cu", "tc_common.cuh", "ptx.cuh", "ptx_pair.cuh"),
                   "tensor"),
    "add_i32": ("add_i32", ("int4.cu",), "hbm"),
    "convert_i4": ("convert_i4_kernel", ("int4.cu",), "hbm"),
    "tc_karatsuba": ("tc_gemm_kernel<3>", ("gemm_tc.cu", "tc_common.cuh", "ptx.cuh"), "tensor"),
    "tc_pair_i16_ahead": ("tc_pair_kernel<2,ahead>", ("gemm_pair.cu", "tc_common.cuh", "ptx.cuh", "ptx_pair.cuh"),
                          "tensor"),
    "conv_rows": ("conv_rows_kernel", ("conv_rows.cu", "tc_common.cuh", "ptx.cuh", "ptx_pair.cuh"), "hbm"),
}
FP8_PER_BF16 = 2.0  # nominal dense fp8 / bf16 tensor rate (4.5 / 2.25 PFLOP/s)
FULL16_RANGE = ("uniform", -32768, 32767)


def parse_args():
    return parse_args_list(None)


def parse_args_list(argv):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=("gemmi", "reference"), default="gemmi")
    p.add_argument("--workload", default="i16_8192", choices=list(gi.WORKLOADS))
    p.add_argument("--no-extra", action="store_true", help="skip the per-workload table")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-sustained", action="store_true", help="skip the two-second back-to-back leg")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU budget of the oracle baseline")
    return p.parse_args(argv)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.file = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [r.split(", ") for r in self.file.read().strip().splitlines() if r.strip()]
        os.unlink(self.file.name)
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
                for nm, v in zip(names, r[4:8]):
                    if v.strip().lower() == "active":
                        reasons.add(nm)
            except (ValueError, IndexError):
                continue
        busy = [s for s in sm if mx and s > 0.3 * max(mx)] or sm
        return {"sm_mhz": statistics.median(busy) if busy else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ helpers
def kernel_source_hash(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2302_07594_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, src_hash: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on this exact kernel source."""
    path = os.path.join(PROFILES, "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f).get(kernel)
    if not d or d.get("source_hash") != src_hash:
        return None
    return d.get("dram_bytes_per_launch")


def workload_bytes(w):
    """Algorithmic HBM bytes of one call: read A, B and C once, write C once (int4 operands packed)."""
    cb = 8 if w.kind == "i16" else 4
    if w.kind == "i4":
        return w.m * ((w.k + 1) // 2) + w.k * ((w.n + 1) // 2) + 2 * w.m * w.n * cb
    op = 2 if w.kind == "i16" else 1
    return w.m * w.k * op + w.k * w.n * op + 2 * w.m * w.n * cb


def max_over_ranks(x: float, world: int, device: str = "cuda") -> float:
    """The largest value of x over all ranks (the slowest replica sets the job's time)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, seconds: float, world: int) -> float:
    """Whole-job rate: every rank processed units_per_rank in the (max-over-ranks) time."""
    return world * units_per_rank / seconds


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# ------------------------------------------------------------------ the oracle (CPU) legs
def oracle_rate(w, seconds: float, threads: int):
    """Times the oracle on a row sample of workload w sized to take about `seconds`."""
    import oracle
    oracle.build()
    _, B, _ = gi.make_inputs(w, rows=slice(0, 1))

    def run(A, C):
        if w.kind == "i4":
            oracle.gemm_i4(gi.pack_nibbles(A), Bp, C, w.k, nthreads=threads)
        else:
            oracle.gemm(A, B, C, nthreads=threads)

    Bp = gi.pack_nibbles(B) if w.kind == "i4" else None
    probe = max(1, min(w.m, threads))
    A, _, C = gi.make_inputs(w, rows=slice(0, probe))
    t0 = time.perf_counter()
    run(A, C)
    t_probe = time.perf_counter() - t0
    per_row = t_probe / probe
    rows = int(max(1, min(w.m, seconds / max(per_row, 1e-9))))
    rows = max(probe, (rows // threads) * threads) if rows >= threads else rows
    A, _, C = gi.make_inputs(w, rows=slice(0, rows))
    t0 = time.perf_counter()
    run(A, C)
    t = time.perf_counter() - t0
    ops = 2 * rows * w.n * w.k
    return ops / t / 1e12, t, rows


def config_of(w, world: int) -> dict:
    """The `config` object of the JSON line; identical in both arms."""
    return {"workload": w.name, "m": w.m, "n": w.n, "k": w.k, "note": w.note,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": f"inputs larger than L2 ({workload_bytes(w) / 2**20:.0f} MiB of A, B, C per step "
                  f"vs {L2_BYTES / 2**20:.0f} MiB L2)"}


def run_reference(args):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    import oracle
    w = gi.WORKLOADS[args.workload]
    threads = oracle.host_cores()
    oracle.build()
    # one step = the oracle on a bounded row sample; the whole run is kept near 90 s of CPU time
    step_s = min(1.5, max(0.05, 90.0 / max(1, args.steps + args.warmup)))
    _, B, _ = gi.make_inputs(w, rows=slice(0, 1))
    if w.kind == "i4":  # the oracle takes the operands in their packed form
        B = gi.pack_nibbles(B)

    def run(A, X):
        if w.kind == "i4":
            oracle.gemm_i4(A, B, X, w.k, nthreads=threads)
        else:
            oracle.gemm(A, B, X, nthreads=threads)

    def rows_of(r):
        A, _, C = gi.make_inputs(w, rows=slice(0, r))
        return (gi.pack_nibbles(A) if w.kind == "i4" else A), C

    A1, C1 = rows_of(min(w.m, threads))
    t0 = time.perf_counter()
    run(A1, C1)
    per_row = (time.perf_counter() - t0) / A1.shape[0]
    rows = int(max(1, min(w.m, step_s / max(per_row, 1e-9))))
    A, C = rows_of(rows)
    for _ in range(args.warmup):
        run(A, C.copy())
    times = []
    for _ in range(args.steps):
        X = C.copy()
        t0 = time.perf_counter()
        run(A, X)
        times.append(time.perf_counter() - t0)
    t = sum(times) / len(times)
    ops = 2 * rows * w.n * w.k
    value = ops / t / 1e12
    sample = f"rows 0..{rows - 1} of {w.m} (full n={w.n}, k={w.k}) per step"
    line = {"metric": {"i16": "int16", "i8": "int8", "i4": "int4"}[w.kind] + " GEMM TOPS (2mnk/s)",
            "value": value, "unit": "TOPS", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": t * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "int64" if w.kind == "i16" else "int32", "data": "synthetic (seeded SplitMix64)",
            "impl": "reference",
            "config": config_of(w, world),
            "cpu_baseline": {"value": value, "unit": "TOPS", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------ the GPU leg
def _time_calls(gm, torch, sets, fn, steps, warmup):
    """(ms per call under CUDA-graph replay, ms per call issued eagerly, kernel timers) of fn(*set),
    rotating over the input sets."""
    nsets = len(sets)
    for i in range(warmup):
        fn(*sets[i % nsets])
    torch.cuda.synchronize()
    gm.kernel_timing(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for i in range(steps):
        fn(*sets[i % nsets])
    e1.record()
    torch.cuda.synchronize()
    eager_ms = e0.elapsed_time(e1) / steps
    kt = {name: gm.kernel_time(kid) for name, kid in gm.KERNELS}
    gm.kernel_timing(False)
    # CUDA-graph replay of the same calls
    ncap = min(steps, 64)
    side = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        for i in range(ncap):
            fn(*sets[i % nsets])
    graph.replay()
    torch.cuda.synchronize()
    reps = max(1, steps // ncap)
    e0.record()
    for _ in range(reps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    graph_ms = e0.elapsed_time(e1) / (reps * ncap)
    assert gm.device_status() == gm.OK
    del graph
    return graph_ms, eager_ms, kt


def time_workload_packed(gm, torch, w, steps, warmup, rotate_bytes=4 * L2_BYTES, max_sets=64):
    """Like time_workload, with B split once per input set (gemmi_pack_b_*, outside the timing) and
    the calls made through gemm_*_packed: weights packed once, activations at run time."""
    per_set = workload_bytes(w)
    nsets = int(min(max_sets, max(1, math.ceil(rotate_bytes / per_set))))
    A, B, C = gi.make_inputs(w)
    sets, packs = [], []
    if w.kind == "i4":
        A, B = gi.pack_nibbles(A), gi.pack_nibbles(B)
        pack = lambda b: gm.pack_b_i4(b, w.n)  # noqa: E731
    else:
        pack = gm.pack_b_i16 if w.kind == "i16" else gm.pack_b_i8
    for _ in range(nsets):
        dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
        pk = pack(dB)
        del dB
        packs.append(pk)
        sets.append((dA, pk, dC))
    torch.cuda.synchronize()
    fn = {"i16": gm.gemm_i16_packed, "i8": gm.gemm_i8_packed, "i4": gm.gemm_i4_packed}[w.kind]
    graph_ms, eager_ms, kt = _time_calls(gm, torch, sets, fn, steps, warmup)
    del sets
    for pk in packs:
        pk.close()
    torch.cuda.empty_cache()
    return graph_ms, eager_ms, kt, nsets


def time_read_floor(gm, torch, w, steps=256, rotate_bytes=4 * L2_BYTES):
    """ms per call of gemmi_stream_read_probe over workload w's B matrices (rotated past L2),
    CUDA-graph replay timed like the GEMM: the skinny kernel's grid, TMA boxes and stage ring
    reading B once and doing nothing else, i.e. the read floor of that kernel."""
    nb = w.k * w.n * 2
    nsets = int(max(1, math.ceil(rotate_bytes / nb)))
    Bs = [torch.zeros((w.k, w.n), dtype=torch.int16, device="cuda") for _ in range(nsets)]
    for b in Bs[:3]:
        gm.stream_read_probe(b)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    ncap = 64
    with torch.cuda.graph(graph, stream=side):
        for i in range(ncap):
            gm.stream_read_probe(Bs[i % nsets], stream=side)
    graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(1, steps // ncap)
    e0.record()
    for _ in range(reps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / (reps * ncap)
    assert gm.device_status() == gm.OK
    del graph, Bs
    torch.cuda.empty_cache()
    return ms


def time_workload(gm, torch, w, steps, warmup, rotate_bytes=4 * L2_BYTES, max_sets=64):
    """Device-resident timing of one workload; rotates input sets so the working set exceeds L2.

    Returns (ms per call under CUDA-graph replay, ms per call issued eagerly, kernel timers, sets).
    The graph replay removes the host's per-call cost (Python, argument checks, launches), which
    is larger than the GPU time of the small workloads.
    """
    per_set = workload_bytes(w)
    nsets = int(min(max_sets, max(1, math.ceil(rotate_bytes / per_set))))
    A, B, C = gi.make_inputs(w)
    if w.kind == "i4":
        A, B = gi.pack_nibbles(A), gi.pack_nibbles(B)
    sets = [tuple(torch.from_numpy(x).cuda() for x in (A, B, C)) for _ in range(nsets)]
    if w.kind == "i4":
        fn = lambda a, b, c: gm.gemm_i4(a, b, c, w.k)  # noqa: E731
    else:
        fn = gm.gemm_i16 if w.kind == "i16" else gm.gemm_i8
    graph_ms, eager_ms, kt = _time_calls(gm, torch, sets, fn, steps, warmup)
    del sets
    torch.cuda.empty_cache()
    return graph_ms, eager_ms, kt, nsets


# The convolution behind the im2col workload, computed from its NHWC activations
# (gemmi_conv2d_i16): batch 32, 56x56, 64 -> 64 channels, 3x3, stride 1, pad 1.
CONV = dict(N=32, H=56, W=56, Cin=64, Cout=64, R=3, S=3, ph=1, pw=1)


def conv_bytes():
    c = CONV
    return (c["N"] * c["H"] * c["W"] * c["Cin"] * 2 + c["R"] * c["S"] * c["Cin"] * c["Cout"] * 2
            + 2 * c["N"] * c["H"] * c["W"] * c["Cout"] * 8)


def time_conv(gm, torch, steps, warmup, rotate_bytes=4 * L2_BYTES):
    """Like time_workload, for the implicit convolution: X with the workload's activation
    distribution (half exact zeros, else [0, 4095]), weights in [-2048, 2047], Y = 0."""
    c = CONV
    nsets = int(max(1, math.ceil(rotate_bytes / conv_bytes())))
    X = gi.half_zero_uniform(1003, (c["N"], c["H"], c["W"], c["Cin"]), 4095, np.int16)
    Wt = gi.uniform_int(1006, (c["R"] * c["S"] * c["Cin"], c["Cout"]), -2048, 2047, np.int16)
    Y = np.zeros((c["N"], c["H"], c["W"], c["Cout"]), np.int64)
    sets = [tuple(torch.from_numpy(x).cuda() for x in (X, Wt, Y)) for _ in range(nsets)]
    fn = lambda x, wt, y: gm.conv2d_i16(x, wt, y, c["R"], c["S"], c["ph"], c["pw"])
    graph_ms, eager_ms, kt = _time_calls(gm, torch, sets, fn, steps, warmup)
    del sets
    torch.cuda.empty_cache()
    return graph_ms, eager_ms, kt, nsets


def int8_tensor_peak(torch):
    """Dense INT8 tensor throughput on this GPU via cuBLASLt (torch._int_mm, 8192^3), in TOPS."""
    try:
        n = 8192
        a = torch.randint(-128, 127, (n, n), dtype=torch.int8, device="cuda")
        b = torch.randint(-128, 127, (n, n), dtype=torch.int8, device="cuda").t()
        for _ in range(3):
            torch._int_mm(a, b)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(10):
            torch._int_mm(a, b)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / 10
        del a, b
        return 2 * n ** 3 / (ms * 1e-3) / 1e12
    except Exception:  # pragma: no cover - reported as unavailable
        return None


# the five workloads of the problem statement, then the extensions, in the compact summary
SUMMARY_ROWS = (("C1", "i16_256", "launch"), ("C2", "i8_4096", "tensor"), ("C3", "conv3x3_im2col", "hbm"),
                ("C4", "i16_8192", "tensor"), ("C5", "skinny_8x4096x4096", "hbm"), ("int4", "i4_8192", "tensor"),
                ("conv", "conv3x3_implicit", "hbm"), ("C4pk", "i16_8192_packed_b", "tensor"),
                ("C2pk", "i8_4096_packed_b", "tensor"), ("C3pk", "conv3x3_im2col_packed_b", "hbm"),
                ("C4ka", "i16_8192_karatsuba", "tensor"), ("C4srs", "i16_8192_srs", "tensor"))


def summarize(extra: dict, peaks: dict) -> dict:
    """One short entry per workload of the per-workload table: microseconds per call (CUDA-graph
    replay), TOPS, GB/s of algorithmic bytes and the fraction of the roofline that bounds it."""
    out = {}
    for key, name, bound in SUMMARY_ROWS:
        e = extra.get(name)
        if not isinstance(e, dict) or "ms" not in e:
            continue
        ent = {"us": round(e["ms"] * 1e3, 1), "TOPS": round(e["TOPS"], 1), "bound": bound}
        if "GB_per_s" in e:
            ent["GBs"] = round(e["GB_per_s"])
        for fk, tag in (("frac_of_fp16_tensor_peak", "fp16"), ("frac_of_fp8_tensor_peak", "fp8"),
                        ("frac_of_limb_tensor_peak", "limb"), ("frac_of_hbm", "hbm"),
                        ("srs_frac_of_hbm", "srs_hbm")):
            if fk in e:
                ent[tag] = round(e[fk], 3)
        fl = e.get("read_floor")
        if isinstance(fl, dict) and "ms" in fl:
            ent["floor_us"] = round(fl["ms"] * 1e3, 2)
        out[key] = ent
    out["peaks"] = {"hbm_GBs": peaks["hbm_gbs"], "bf16_TFs": peaks["bf16_tflops"], "src": peaks["source"]}
    return out


def run_gemmi(args):
    import torch
    import torch.distributed as dist

    import paper_2302_07594_gb300 as gm

    world, rank, local = dist_setup()
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    gm.lib()
    peaks = measured_peaks()
    w = gi.WORKLOADS[args.workload]
    A, B, C = gi.make_inputs(w)
    if w.kind == "i4":  # the int4 operands travel packed, two values to a byte
        A, B = gi.pack_nibbles(A), gi.pack_nibbles(B)
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    if w.kind == "i4":
        fn = lambda a, b, c: gm.gemm_i4(a, b, c, w.k)  # noqa: E731
    else:
        fn = gm.gemm_i16 if w.kind == "i16" else gm.gemm_i8
    for _ in range(args.warmup):
        fn(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK

    # ---- timed region: K steps, device-resident inputs (the working set is larger than L2)
    sampler = ClockSampler(local)
    sampler.start()
    gm.kernel_timing(True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        fn(dA, dB, dC)
    e1.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms = e0.elapsed_time(e1) / args.steps
    kt = {name: gm.kernel_time(kid) for name, kid in gm.KERNELS}
    gm.kernel_timing(False)
    assert gm.device_status() == gm.OK
    ms = max_over_ranks(ms, world)
    value = job_throughput(w.ops, ms * 1e-3, world) / 1e12

    # ---- dominant kernel (most device time in the timed region) and its roofline
    launches = sum(kn for _, kn in kt.values())
    kname = max((name for name in KERNEL_INFO if kt[name][1] > 0), key=lambda name: kt[name][0])
    sym, src, bound = KERNEL_INFO[kname]
    kms, kn = kt[kname]
    per_launch_ms = kms / max(kn, 1)
    if bound == "tensor" and w.kind == "i16":
        achieved = w.ops / (per_launch_ms * 1e-3) / 1e12
        peak = peaks["bf16_tflops"] / 4.0
        roof = {"bound": "tensor", "kernel": sym, "achieved": achieved, "peak": peak, "unit": "TOPS",
                "frac": achieved / peak,
                "peak_note": f"fp16 dense tensor peak ({peaks['source']} bf16 burst {peaks['bf16_tflops']} TFLOP/s, "
                             "fp16 = bf16 rate) / 4 limb products per int16 multiply-add",
                "frac_of_sustained": achieved / (peaks["bf16_tflops_sustained"] / 4.0),
                "kernel_ms": per_launch_ms}
    elif bound == "tensor" and w.kind == "i4":
        achieved = w.ops / (per_launch_ms * 1e-3) / 1e12
        peak = peaks["bf16_tflops"] * FP8_PER_BF16
        roof = {"bound": "tensor", "kernel": sym, "achieved": achieved, "peak": peak, "unit": "TOPS",
                "frac": achieved / peak,
                "peak_note": f"fp8 dense tensor peak: {peaks['source']} bf16 burst {peaks['bf16_tflops']} TFLOP/s x "
                             f"{FP8_PER_BF16} (nominal fp8 / bf16 rate); one E4M3 product per int4 multiply-add",
                "kernel_ms": per_launch_ms}
    elif bound == "tensor":
        achieved = w.ops / (per_launch_ms * 1e-3) / 1e12
        peak = peaks["bf16_tflops"]
        roof = {"bound": "tensor", "kernel": sym, "achieved": achieved, "peak": peak, "unit": "TOPS",
                "frac": achieved / peak, "peak_note": "fp16 dense tensor peak (one fp16 product per int8 product)",
                "kernel_ms": per_launch_ms}
    else:
        achieved = workload_bytes(w) / (per_launch_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": sym, "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"], "kernel_ms": per_launch_ms}
    src_hash = kernel_source_hash(src)
    traffic = recorded_traffic(sym, src_hash)
    roof["traffic"] = traffic
    roof["source_hash"] = src_hash
    roof["peak_source"] = peaks["source"]

    # ---- the same call back to back for about two seconds (not the timed region): the tensor-bound
    # kernels reach the board's power cap within a fraction of a second and the SM clock settles
    # below its maximum; this figure and its clock sit beside the short timed region's
    sustained = None
    if rank == 0 and not args.no_sustained:
        n_sus = max(1, min(5000, int(2000.0 / max(ms, 1e-3))))
        sampler = ClockSampler(local)
        sampler.start()
        e0.record()
        for _ in range(n_sus):
            fn(dA, dB, dC)
        e1.record()
        torch.cuda.synchronize()
        sclk = sampler.stop()
        sms = e0.elapsed_time(e1) / n_sus
        sustained = {"ms_per_step": sms, "value": w.ops / (sms * 1e-3) / 1e12, "unit": "TOPS", "steps": n_sus,
                     "sm_mhz": sclk["sm_mhz"], "reasons": sclk["reasons"],
                     "what": "the timed call back to back for about 2 s (at most 5000 calls) after the timed region"}
        assert gm.device_status() == gm.OK

    int8_peak = int8_tensor_peak(torch)

    # ---- end to end through the host-buffer C ABI (copies inside the timed region)
    op_t = {"i16": torch.int16, "i8": torch.int8, "i4": torch.uint8}[w.kind]
    c_t = torch.int64 if w.kind == "i16" else torch.int32
    hA = torch.empty(A.shape, dtype=op_t, pin_memory=True).numpy()
    hB = torch.empty(B.shape, dtype=op_t, pin_memory=True).numpy()
    hC = torch.empty(C.shape, dtype=c_t, pin_memory=True).numpy()
    hA[...] = A
    hB[...] = B
    hC[...] = C
    if w.kind == "i4":
        host_fn = lambda a, b, c: gm.gemm_i4_host(a, b, c, w.k)  # noqa: E731
    else:
        host_fn = gm.gemm_i16_host if w.kind == "i16" else gm.gemm_i8_host
    gm.set_stream(torch.cuda.current_stream())
    # warm-up calls as for the device-resident leg (the first host-path call of a process sets up
    # its staging buffers and streams); the timed loop is long enough (up to 60 calls, about
    # 0.3 s at 8192^3) that an occasional host-side stall of a few tens of ms weighs little
    for _ in range(max(3, min(args.warmup, 5))):
        host_fn(hA, hB, hC)
    e2e_steps = max(3, min(args.steps, 60))
    if world > 1:
        dist.barrier()
    # each call returns after its results are in host memory, so the calls are timed one by one as
    # well: the mean over all of them is the figure, the median shows it without the occasional
    # host-side stalls of tens of milliseconds that plain pinned copies of the same size see too
    per_call = []
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        tc = time.perf_counter()
        host_fn(hA, hB, hC)
        per_call.append(time.perf_counter() - tc)
    e2e_s = (time.perf_counter() - t0) / e2e_steps
    e2e_s = max_over_ranks(e2e_s, world)
    med_s = max_over_ranks(statistics.median(per_call), world)
    e2e = {"value": job_throughput(w.ops, e2e_s, world) / 1e12, "unit": "TOPS", "ms_per_step": e2e_s * 1e3,
           "h2d_bytes_per_step": int(A.nbytes + B.nbytes + C.nbytes), "d2h_bytes_per_step": int(C.nbytes),
           "steps": e2e_steps, "warmup": max(3, min(args.warmup, 5)), "api": f"gemm_{w.kind}_host",
           "median_ms_per_call": med_s * 1e3, "median_value": job_throughput(w.ops, med_s, world) / 1e12,
           "calls_over_1.5x_median": sum(1 for x in per_call if x > 1.5 * statistics.median(per_call))}
    del hA, hB, hC

    # ---- per-workload table (each workload's own bound), rank 0 only
    extra = {}
    if rank == 0 and not args.no_extra:
        del dA, dB, dC
        torch.cuda.empty_cache()
        for name, ow in gi.WORKLOADS.items():
            try:
                oms, eager_ms, okt, nsets = time_workload(gm, torch, ow, steps=30 if ow.ops > 1e11 else 128, warmup=5)
            except Exception as ex:  # pragma: no cover
                extra[name] = {"error": str(ex)}
                continue
            ent = {"ms": oms, "timing": "CUDA-graph replay, per call", "eager_ms": eager_ms,
                   "TOPS": ow.ops / (oms * 1e-3) / 1e12,
                   "GB_per_s": workload_bytes(ow) / (oms * 1e-3) / 1e9, "input_sets_rotated": nsets}
            ent["kernel_ms"] = {KERNEL_INFO[name][0]: okt[name][0] / okt[name][1]
                                for name in KERNEL_INFO if okt[name][1] > 0}
            if ow.kind == "i8":
                ent["frac_of_fp16_tensor_peak"] = ent["TOPS"] / peaks["bf16_tflops"]
            elif ow.kind == "i4":
                ent["frac_of_fp8_tensor_peak"] = ent["TOPS"] / (peaks["bf16_tflops"] * FP8_PER_BF16)
                ent["fp8_peak_note"] = (f"bf16 burst {peaks['bf16_tflops']} TFLOP/s ({peaks['source']}) x "
                                        f"{FP8_PER_BF16} (nominal fp8 / bf16 dense rate)")
            else:
                ent["frac_of_limb_tensor_peak"] = ent["TOPS"] / (peaks["bf16_tflops"] / 4)
                ent["frac_of_hbm"] = ent["GB_per_s"] / peaks["hbm_gbs"]
            if int8_peak and ow.kind != "i4":
                ent["frac_of_int8_roofline_div4" if ow.kind == "i16" else "frac_of_int8_roofline"] = (
                    ent["TOPS"] / (int8_peak / 4 if ow.kind == "i16" else int8_peak))
            if name.startswith("skinny"):
                # the per-call floor: the same grid, TMA boxes and stage ring reading the same
                # rotating B matrices once, with no arithmetic (gemmi_stream_read_probe)
                try:
                    fms = time_read_floor(gm, torch, ow)
                    fgbs = ow.k * ow.n * 2 / (fms * 1e-3) / 1e9
                    ent["read_floor"] = {"what": "gemmi_stream_read_probe: B streamed as the skinny kernel "
                                                 "streams it, nothing computed; CUDA-graph replay",
                                         "ms": fms, "GB_per_s": fgbs, "frac_of_hbm": fgbs / peaks["hbm_gbs"]}
                except Exception as ex:  # pragma: no cover
                    ent["read_floor"] = {"error": str(ex)}
            extra[name] = ent
        # the same calls with the weights split once (gemmi_pack_b_*): the operand split then covers
        # A only, and the narrow-n kernel has no split at all
        for name in ("i16_8192", "i8_4096", "conv3x3_im2col", "i4_8192"):
            ow = gi.WORKLOADS[name]
            try:
                oms, eager_ms, okt, nsets = time_workload_packed(gm, torch, ow, steps=30 if ow.ops > 1e11 else 128,
                                                                 warmup=5)
            except Exception as ex:  # pragma: no cover
                extra[name + "_packed_b"] = {"error": str(ex)}
                continue
            ent = {"ms": oms, "timing": "CUDA-graph replay, per call; B packed once outside the timing",
                   "eager_ms": eager_ms, "TOPS": ow.ops / (oms * 1e-3) / 1e12, "input_sets_rotated": nsets,
                   "kernel_ms": {KERNEL_INFO[k][0]: okt[k][0] / okt[k][1] for k in KERNEL_INFO if okt[k][1] > 0}}
            if ow.kind == "i8":
                ent["frac_of_fp16_tensor_peak"] = ent["TOPS"] / peaks["bf16_tflops"]
            elif ow.kind == "i4":
                ent["frac_of_fp8_tensor_peak"] = ent["TOPS"] / (peaks["bf16_tflops"] * FP8_PER_BF16)
            else:
                ent["frac_of_limb_tensor_peak"] = ent["TOPS"] / (peaks["bf16_tflops"] / 4)
            extra[name + "_packed_b"] = ent
        # Karatsuba's three limb products (GEMMI_OPT_KARATSUBA) against the four-product default, at
        # int16 8192^3: the call and its kernels (the sum planes are timed with the split)
        try:
            ow = gi.WORKLOADS["i16_8192"]
            gm.set_option(gm.OPT_KARATSUBA, 1)
            try:
                oms, eager_ms, okt, nsets = time_workload(gm, torch, ow, steps=20, warmup=3)
            finally:
                gm.set_option(gm.OPT_KARATSUBA, 0)
            kms = {KERNEL_INFO[k][0]: okt[k][0] / okt[k][1] for k in KERNEL_INFO if okt[k][1] > 0}
            kk = kms.get(KERNEL_INFO["tc_karatsuba"][0])
            extra["i16_8192_karatsuba"] = {
                "ms": oms, "timing": "CUDA-graph replay, per call", "eager_ms": eager_ms,
                "TOPS": ow.ops / (oms * 1e-3) / 1e12, "kernel_ms": kms,
                "kernel_TOPS": (ow.ops / (kk * 1e-3) / 1e12) if kk else None,
                "what": "int16 8192^3 with three limb products (HH, LL, (h_a+l_a)(h_b+l_b)) on one SM per tile"}
        except Exception as ex:  # pragma: no cover
            extra["i16_8192_karatsuba"] = {"error": str(ex)}
        # the requantising output (NEXT-3): int16 C += srs(A*B, 16) on the int16 8192^3 operands; the
        # exact sums go to an int64 scratch, then one pass shifts, rounds, saturates and adds
        try:
            ow = gi.WORKLOADS["i16_8192"]
            A16, B16, _ = gi.make_inputs(ow)
            sset = [(torch.from_numpy(A16).cuda(), torch.from_numpy(B16).cuda(),
                     torch.zeros((ow.m, ow.n), dtype=torch.int16, device="cuda"))]
            oms, eager_ms, okt = _time_calls(gm, torch, sset, lambda a, b, c: gm.gemm_i16_srs(a, b, c, 16), 20, 3)
            del sset
            torch.cuda.empty_cache()
            kms = {KERNEL_INFO[k][0]: okt[k][0] / okt[k][1] for k in KERNEL_INFO if okt[k][1] > 0}
            srs_ms = kms.get(KERNEL_INFO["srs"][0])
            srs_bytes = 12 * ow.m * ow.n  # the int64 sums read, the int16 C read and written
            ent = {"ms": oms, "timing": "CUDA-graph replay, per call", "eager_ms": eager_ms,
                   "TOPS": ow.ops / (oms * 1e-3) / 1e12, "kernel_ms": kms,
                   "what": "gemm_i16_srs, shift 16, on the int16 8192^3 operands: exact sums into an int64 "
                           "scratch (zeroed, then the GEMM), then one shift-round-saturate-add pass into int16 C"}
            if srs_ms:
                ent["srs_GB_per_s"] = srs_bytes / (srs_ms * 1e-3) / 1e9
                ent["srs_frac_of_hbm"] = ent["srs_GB_per_s"] / peaks["hbm_gbs"]
            extra["i16_8192_srs"] = ent
        except Exception as ex:  # pragma: no cover
            extra["i16_8192_srs"] = {"error": str(ex)}
        # the precision sweep at equal sizes: int16 at 4096^3, int8 at 8192^3 and int4 at 4096^3
        # beside the table's int16 / int4 8192^3 and int8 4096^3 (same value distributions)
        sweep = {}
        for sw in (gi.Workload("i16_4096", "i16", 4096, 4096, 4096, 1010, FULL16_RANGE, FULL16_RANGE, ("zero",),
                               "int16 GEMM 4096^3"),
                   gi.Workload("i8_8192", "i8", 8192, 8192, 8192, 1008, ("uniform", -128, 127),
                               ("uniform", -128, 127), ("zero",), "int8 GEMM 8192^3"),
                   gi.Workload("i4_4096", "i4", 4096, 4096, 4096, 1009, ("uniform", -8, 7), ("uniform", -8, 7),
                               ("zero",), "int4 GEMM 4096^3")):
            try:
                sms, seager, skt, sn = time_workload(gm, torch, sw, steps=30, warmup=5)
            except Exception as ex:  # pragma: no cover
                sweep[sw.name] = {"error": str(ex)}
                continue
            sweep[sw.name] = {"ms": sms, "timing": "CUDA-graph replay, per call", "eager_ms": seager,
                              "TOPS": sw.ops / (sms * 1e-3) / 1e12, "input_sets_rotated": sn,
                              "kernel_ms": {KERNEL_INFO[k][0]: skt[k][0] / skt[k][1] for k in KERNEL_INFO
                                            if skt[k][1] > 0}}
        extra["precision_sweep"] = sweep
        try:
            cms, ceager, ckt, cn = time_conv(gm, torch, steps=128, warmup=5)
            ops = 2 * CONV["N"] * CONV["H"] * CONV["W"] * CONV["Cout"] * CONV["R"] * CONV["S"] * CONV["Cin"]
            extra["conv3x3_implicit"] = {
                "ms": cms, "timing": "CUDA-graph replay, per call", "eager_ms": ceager,
                "what": "gemmi_conv2d_i16 on NHWC activations: the im2col workload's convolution "
                        "without forming the lowered matrix", "shape": CONV,
                "TOPS": ops / (cms * 1e-3) / 1e12, "GB_per_s": conv_bytes() / (cms * 1e-3) / 1e9,
                "frac_of_hbm": conv_bytes() / (cms * 1e-3) / 1e9 / peaks["hbm_gbs"], "input_sets_rotated": cn,
                "kernel_ms": {KERNEL_INFO[k][0]: ckt[k][0] / ckt[k][1] for k in KERNEL_INFO if ckt[k][1] > 0}}
        except Exception as ex:  # pragma: no cover
            extra["conv3x3_implicit"] = {"error": str(ex)}

    # ---- CPU baseline: the oracle on a bounded sample (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        cores = oracle.host_cores()
        v, t, rows = oracle_rate(w, args.cpu_seconds, cores)
        cpu = {"value": v, "unit": "TOPS", "cores": cores, "kind": "oracle",
               "sample": f"rows 0..{rows - 1} of {w.m} (full n={w.n}, k={w.k}), {t:.1f} s on {cores} threads"}
        # the two small workloads whole, on one thread (the oracle's plain loop, for scale)
        single = {}
        for sname in ("i16_256", "skinny_8x4096x4096"):
            sw = gi.WORKLOADS[sname]
            sA, sB, sC = gi.make_inputs(sw)
            t0 = time.perf_counter()
            oracle.gemm(sA, sB, sC, nthreads=1)
            st = time.perf_counter() - t0
            single[sname] = {"ms": st * 1e3, "TOPS": sw.ops / st / 1e12, "threads": 1}
        cpu["single_thread_whole_workloads"] = single

    if rank == 0:
        line = {
            "metric": {"i16": "int16", "i8": "int8", "i4": "int4"}[w.kind] + " GEMM TOPS (2mnk/s)",
            "value": value, "unit": "TOPS", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "int64" if w.kind == "i16" else "int32",
            "data": "synthetic (seeded SplitMix64 inputs of the workload's shape and value distribution)",
            "config": config_of(w, world),
            "roofline": roof,
            "int8_roofline": None if int8_peak is None else {
                "int8_tensor_tops": int8_peak, "how": "torch._int_mm (cuBLASLt) 8192^3 on this GPU",
                "effective_int16_peak": int8_peak / 4,
                "frac": (roof["achieved"] / (int8_peak / 4)) if roof["unit"] == "TOPS" and w.kind == "i16" else None,
                "note": "fp16 limb products on tcgen05 run far above the legacy INT8 path, so this "
                        "fraction exceeds 1; it is not an efficiency figure"},
            "e2e": e2e,
            "gpu_launches": int(launches),
            "clocks": clocks,
            "cpu_baseline": cpu,
            "sustained": sustained,
            "workloads": extra,
            "summary": summarize(extra, peaks),
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_gemmi(args)


if __name__ == "__main__":
    sys.exit(main())
