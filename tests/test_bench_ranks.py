"""bench.py's multi-GPU path is replicas only: every rank runs the whole
workload on its own GPU and nothing is exchanged but the timing. Its rank
logic (barrier, max over ranks, whole-job rate, rank-0-only reference arm)
runs here on CPU with world_size-2 gloo process groups."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dev = torch.device("cpu")
        bench.dist_barrier(world, dev)
        slowest = bench.max_over_ranks(10.0 + rank, world, dev)      # rank 1 is the slow one
        rate = bench.whole_job_rate(world, 1000, 8, slowest)
        out.put((rank, slowest, rate))
        bench.dist_barrier(world, dev)
    finally:
        dist.destroy_process_group()


def test_replicas_max_over_ranks_gloo():
    world, port = 2, free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [11.0, 11.0]          # every rank sees the slowest time
    assert res[0][2] == pytest.approx(2 * 1000 * 8 / 11.0 / 1e9)   # units of all ranks / that time


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1, torch.device("cpu")) == 3.5
    assert bench.whole_job_rate(1, 2, 3, 1.0) == pytest.approx(6e-9)


def test_reference_arm_runs_on_rank0_only(capsys, monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    bench.run_reference(bench.parse_args())
    assert capsys.readouterr().out == ""


def test_reference_arm_line_on_cpu(capsys, monkeypatch):
    """Rank 0's reference arm (the oracle on the host cores) prints one JSON
    line with the contract's keys, on a machine without a GPU."""
    import json
    monkeypatch.delenv("RANK", raising=False)
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--config", "opt-1.3b", "--steps", "1",
                                      "--warmup", "1", "--cpu-seconds", "0.4", "--cpu-workers", "2"])
    bench.run_reference(bench.parse_args())
    lines = [ln for ln in capsys.readouterr().out.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    for key in ("metric", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "scaling", "dtype", "data", "config"):
        assert key in d, key
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_small_workload_on_cpu(capsys, monkeypatch):
    """--config tiny --impl reference runs the oracle's full steps on the
    whole small workload (split over host processes) and prints one line."""
    monkeypatch.setenv("RANK", "0")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--config", "tiny", "--steps", "1",
                                      "--cpu-workers", "2"])
    bench.main()
    import json
    d = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["value"] > 0 and d["config"]["d"] == 1 << 20
    assert d["cpu_baseline"]["cores"] == 2 and d["e2e"]["value"] == d["value"]


def test_cpu_model_and_single_thread_oracle():
    assert isinstance(bench.cpu_model(), str) and bench.cpu_model()
    ps = bench.W.OPT_1_3B
    v, n = bench.time_oracle_single(ps, 0.2)
    assert v > 0 and n % 16 == 0 and n >= 16
