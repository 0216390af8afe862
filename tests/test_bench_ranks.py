"""The multi-rank logic of bench.py on CPU: two gloo ranks (127.0.0.1) agree
on the slowest rank's step time, the whole-job value counts every rank's
positions, and the reference arm does its work on rank 0 only."""
import importlib.util
import os
import socket

import pytest

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b = _bench()
        t = b.max_over_ranks(1.5 + rank, world, "cpu")  # rank 1 is the slow one
        out[rank] = (t, b.replicas_value(32, world, t / 1000.0))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_step():
    import torch.multiprocessing as mp
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    assert out[0] == out[1]
    t, v = out[0]
    assert t == 2.5
    assert abs(v - 32 * 2 / 2.5e-3) < 1e-6


def test_single_rank_is_a_no_op():
    b = _bench()
    assert b.max_over_ranks(3.25, 1, "cpu") == 3.25
    assert b.replicas_value(32, 1, 0.5) == 64.0


def test_reference_arm_only_on_rank_zero(capsys):
    b = _bench()

    class Args:
        config, state, steps, warmup = "tiny", "select", 1, 0

    b.run_reference(Args(), rank=1, world=2)  # returns at once, prints nothing
    assert capsys.readouterr().out == ""


def test_reference_arm_json_contract():
    """bench.py --impl reference prints one JSON line with the contract's keys
    (the tiny config, one step of the CPU oracle)."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--config", "tiny", "--steps", "1", "--warmup", "1"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["warmup"] >= 3
    assert d["value"] > 0 and d["config"]["workload"]
    for k in ("value", "unit", "cores", "kind", "sample"):
        assert k in d["cpu_baseline"], k
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    for k in ("value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step"):
        assert k in d["e2e"], k
