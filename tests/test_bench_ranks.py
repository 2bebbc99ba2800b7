"""bench.py's rank logic on CPU with world_size-2 gloo process groups: the
default multi-GPU path (replicas: every rank runs the whole workload on its
own GPU, only the timing is exchanged -- barrier, max over ranks, whole-job
rate, rank-0-only reference arm) and the --probe-parallel step (probe k on
rank k mod R, the loss table all-gathered, every rank updating), the latter
with the oracle as each rank's arithmetic."""
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
    # the same config dict as the device arm prints (built by the same function)
    args = bench.parse_args()
    assert d["config"] == bench.stream_config(bench.param_set(args), args, 1)
    assert d["config"]["workload"] == "opt-1.3b-shape-bf16" and d["config"]["tensors"] == 388


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
    args = bench.parse_args()
    assert d["config"] == bench.tiny_config(bench.param_set(args), args, 1)


def test_cpu_model_and_single_thread_oracle():
    assert isinstance(bench.cpu_model(), str) and bench.cpu_model()
    ps = bench.W.OPT_1_3B
    v, n = bench.time_oracle_single(ps, 0.2)
    assert v > 0 and n % 16 == 0 and n >= 16


# ------------------------------------------- --probe-parallel, oracle arithmetic
def pp_worker(rank, world, port, out):
    """One rank of bench.py's probe-parallel step with the oracle as the
    arithmetic: out-of-place pair passes of its probes on host copies, the
    loss rows all-gathered over gloo, the oracle's preconditioner and update."""
    import numpy as np

    import oracle
    from paper_2609_38095_gb300 import replicas as R
    from paper_2609_38095_gb300 import workloads as W
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    if world > 1:
        dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dts = [W.DT_BF16, W.DT_F32]
        rng = np.random.default_rng(5)
        theta = [W.random_storage(rng, n, dt) for n, dt in zip([1000, 333], dts)]
        K, eps, seed = 7, 1e-3, W.step_seed(9)
        L = torch.from_numpy(W.synthetic_losses(K, 9))
        passes = []

        def pair_pass(k):
            plus, minus = [t.copy() for t in theta], [t.copy() for t in theta]
            oracle.perturb(plus, dts, seed, k, eps)
            oracle.perturb(minus, dts, seed, k, -eps)
            passes.append(k)

        def finish(table):
            rc, c, _, _ = oracle.precondition(table.numpy(), eps)
            assert rc == oracle.OK
            oracle.update(theta, dts, seed, c, eps)

        table = bench.probe_parallel_step(L, K, rank, world, pair_pass, lambda rows: R.all_gather_losses(rows, K),
                                          finish)
        out.put((rank, passes, table.numpy(), [t.copy() for t in theta]))
    finally:
        if world > 1:
            dist.destroy_process_group()


def run_pp(world):
    port = free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=pp_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=300) for _ in range(world)), key=lambda x: x[0])
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    return res


def test_probe_parallel_step_gloo_two_ranks():
    """Two gloo ranks split the probes (0, 2, 4, 6 and 1, 3, 5), both end up
    with the full seeded loss table and with the same weights, bit for bit
    those of one process running every probe."""
    import numpy as np
    from paper_2609_38095_gb300 import workloads as W
    two = run_pp(2)
    one = run_pp(1)
    assert two[0][1] == [0, 2, 4, 6] and two[1][1] == [1, 3, 5] and one[0][1] == list(range(7))
    want = W.synthetic_losses(7, 9)
    for _, _, table, _ in two + one:
        np.testing.assert_array_equal(table, want)
    for r in range(2):
        for a, b in zip(two[r][3], one[0][3]):
            view = np.uint32 if a.dtype == np.float32 else np.uint16
            np.testing.assert_array_equal(a.view(view), b.view(view))


def test_schedule_defaults_and_combinations(monkeypatch):
    """The parameter sets default to the fused schedule and the small
    workload to onepass; onepass needs --config tiny, which does not run the
    pair schedule."""
    for argv, want in ((["bench.py"], "fused"), (["bench.py", "--config", "tiny"], "onepass"),
                       (["bench.py", "--config", "tiny", "--schedule", "fused"], "fused"),
                       (["bench.py", "--config", "opt-1.3b", "--schedule", "alg1"], "alg1")):
        monkeypatch.setattr(sys, "argv", argv)
        assert bench.parse_args().schedule == want, argv
    for argv in (["bench.py", "--schedule", "onepass"], ["bench.py", "--config", "tiny", "--schedule", "pair"]):
        monkeypatch.setattr(sys, "argv", argv)
        with pytest.raises(SystemExit):
            bench.parse_args()
