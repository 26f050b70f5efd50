"""The multi-GPU mode of bench.py is replicas only: every rank runs the whole workload, and the
job's time is the slowest rank's.  Its host-side logic runs here as two gloo ranks on the CPU
(no GPU): the max-over-ranks reduction, the whole-job rate and the rank handling of the
reference arm."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method="env://", rank=rank, world_size=world)
    try:
        assert bench.dist_setup() == (world, rank, rank)
        local_ms = [2.0, 3.5, 1.25][rank]
        ms = bench.max_over_ranks(local_ms, world, device="cpu")
        value = bench.job_throughput(1.0e9, ms * 1e-3, world)
        dist.barrier()
        out[rank] = (ms, value)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_replicas_take_the_slowest_rank(world):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        slowest = max([2.0, 3.5, 1.25][:world])
        for r in range(world):
            ms, value = out[r]
            assert ms == slowest
            assert value == pytest.approx(world * 1.0e9 / (slowest * 1e-3))


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(4.5, 1) == 4.5
    assert bench.job_throughput(10.0, 2.0, 1) == 5.0


def test_reference_arm_runs_on_rank_0_only(monkeypatch):
    # the other ranks of a torchrun reference arm exit 0 without work or output
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = bench.parse_args_list(["--impl", "reference", "--steps", "1", "--warmup", "0"])
    assert bench.run_reference(args) == 0


@pytest.mark.parametrize("workload", ["i16_256", "i4_8192"])
def test_reference_arm_prints_one_json_line(workload):
    # the reference arm is the CPU oracle on bounded row samples: it runs here, without a GPU
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload", workload,
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=600,
                       env={**os.environ, "RANK": "0", "WORLD_SIZE": "1"})
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["steps"] == 2 and d["warmup"] == 1
    assert d["metric"].startswith({"i16_256": "int16", "i4_8192": "int4"}[workload])
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["config"]["workload"] == workload
