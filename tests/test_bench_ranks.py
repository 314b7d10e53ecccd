"""The multi-rank path of bench.py on the CPU: two gloo ranks agree on the max
of their step times and on the whole-job throughput, and the reference arm
runs on rank 0 only (the others exit at once)."""
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


def _worker(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    # rank r reports step 1 + r ms, e2e 3 + r ms, attention 0.5 + r ms; 80 rows per step
    agg = bench.aggregate_over_ranks(1.0 + rank, 3.0 + rank, 0.5 + rank, 80, world)
    out.put((rank, agg))
    dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_max():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        agg = res[r]
        assert agg["step_ms"] == 2.0 and agg["e2e_ms"] == 4.0 and agg["attn_ms"] == 1.5
        assert agg["value"] == 2 * 80 / 2e-3 and agg["e2e_value"] == 2 * 80 / 4e-3


def _remeasure_worker(rank, world, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    import bench
    from test_bench_clocks import GOOD, THERMAL, FakeClock
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    runs = []

    def region():
        runs.append(1)
        return len(runs)

    def max_over_ranks(x):
        t = torch.tensor([x], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    # only rank 1 sees a thermal slowdown; both ranks must run the region again
    records = [THERMAL, GOOD] if rank == 1 else [GOOD, GOOD]
    res, clocks, again = bench.measure_with_clock_check(region, lambda: None, FakeClock(records),
                                                        barrier=dist.barrier, allreduce_max=max_over_ranks)
    out.put((rank, len(runs), again))
    dist.destroy_process_group()


def test_a_bad_clock_on_one_rank_remeasures_every_rank():
    pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_remeasure_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict((r, (n, a)) for r, n, a in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res == {0: (2, True), 1: (2, True)}


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    agg = bench.aggregate_over_ranks(2.0, 5.0, 1.0, 80, 1)
    assert agg["value"] == 80 / 2e-3 and agg["attn_ms"] == 1.0


def _reference(rank, world):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus",
                           str(world), "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                          text=True, timeout=300, cwd=ROOT)


def test_reference_arm_runs_on_rank_zero_only():
    r1 = _reference(1, 2)
    assert r1.returncode == 0 and r1.stdout.strip() == ""
    r0 = _reference(0, 2)
    assert r0.returncode == 0, r0.stderr[-2000:]
    line = json.loads(r0.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["n_gpus"] == 2
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"
