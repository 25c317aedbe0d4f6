"""Host logic of bench.py's multi-process path, on CPU with the gloo backend.

Under torchrun every rank times its own replica of the workload; the job's time
is the slowest rank's (an all-reduce MAX) and the reported value counts the
units of all ranks.  Two gloo ranks on 127.0.0.1 run the same helpers that the
GPU bench runs over NCCL, and the reference arm must stay silent on ranks > 0.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, q):
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(times[rank], dist, torch.device("cpu"))
        value = bench.job_throughput(1000, world, 10, ms)
        q.put((rank, ms, value))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    world, times = 2, [12.5, 40.25]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, times, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(world))
    for rank, ms, value in res:
        assert ms == max(times)
        # 1000 units per rank per step, 2 ranks, 10 steps in 40.25 ms
        assert value == pytest.approx(1000 * 2 * 10 / (40.25 / 1e3))


def test_one_process_needs_no_group():
    assert bench.max_over_ranks(3.0, None, None) == 3.0
    assert bench.job_throughput(65536, 1, 20, 7.5) == pytest.approx(65536 * 20 / 7.5e-3)


def test_reference_arm_is_silent_off_rank_zero(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1"])
    bench.main()
    assert capsys.readouterr().out == ""


def test_cpu_list_parsing():
    assert bench._cpulist("0-3,8-11,16\n") == {0, 1, 2, 3, 8, 9, 10, 11, 16}
    assert bench._cpulist("5") == {5}
    assert bench._cpulist("") == set()


def test_near_gpu_host_is_best_effort_and_restores_affinity():
    """Without a device (or its sysfs entry) the NUMA pinning is skipped; the thread's CPU
    affinity is the same after the block as before it."""
    before = os.sched_getaffinity(0)
    with bench.NearGpuHost(0) as host:
        pass
    assert os.sched_getaffinity(0) == before
    assert host.cpus == 0 or host.node is not None


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` (the oracle, on the host cores) prints one JSON line with
    the contract's keys, the same metric and workload as the GPU arm, and the e2e object."""
    import json
    import subprocess
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert p.returncode == 0, p.stderr
    lines = [ln for ln in p.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["steps"] == 1
    assert d["config"]["workload"] == bench.WORKLOAD and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
