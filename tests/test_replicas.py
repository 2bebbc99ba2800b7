"""The probe-parallel step over replicas (Sec. 4.3, Algorithm 1, with the
loss exchange as an all-gather and every replica updating).

CPU: the probe partition, the table assembly, and whole steps on world-size
2 and 3 gloo process groups with the oracle doing each rank's arithmetic;
every rank must end with the same table and the same parameters as one
process doing all K probes. GPU: the library's step as one replica, and
three replicas simulated one after the other on one device (no kernel waits
on another), against the one-replica step and the oracle."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2609_38095_gb300 import replicas as R
from paper_2609_38095_gb300 import workloads as W

from gpu_helpers import assert_update_close, storage_bits


# ----------------------------------------------------------------- host logic
@pytest.mark.parametrize("K", [0, 1, 7, 8, 64, 257])
@pytest.mark.parametrize("world", [1, 2, 3, 8])
def test_probes_partition(K, world):
    owned = [list(R.probes_of_rank(K, r, world)) for r in range(world)]
    flat = sorted(k for o in owned for k in o)
    assert flat == list(range(K))                      # every probe once
    assert all(k % world == r for r, o in enumerate(owned) for k in o)
    assert max(len(o) for o in owned) - min(len(o) for o in owned) <= 1


def test_probes_of_rank_rejects_bad_rank():
    for rank, world in ((2, 2), (-1, 2), (0, 0)):
        with pytest.raises(ValueError):
            R.probes_of_rank(8, rank, world)


@pytest.mark.parametrize("K,world", [(7, 3), (8, 2), (2, 4), (0, 2)])
def test_assemble_losses_places_rows(K, world):
    m = -(-K // world)
    full = torch.arange(K * 3, dtype=torch.float64).reshape(K, 3) + 0.5
    parts = []
    for r in range(world):
        mine = list(R.probes_of_rank(K, r, world))
        p = torch.full((m, 3), float("nan"), dtype=torch.float64)   # padding must be ignored
        p[:len(mine)] = full[mine]
        parts.append(p)
    assert torch.equal(R.assemble_losses(parts, K, world), full)
    with pytest.raises(ValueError):
        R.assemble_losses(parts[:-1], K, world)


def test_all_gather_losses_single_process_checks_shape():
    own = torch.zeros(5, 3, dtype=torch.float64)
    assert torch.equal(R.all_gather_losses(own, 5), own)
    with pytest.raises(ValueError):
        R.all_gather_losses(own, 6)


# ----------------------------------------------- gloo ranks, oracle arithmetic
DTS = [W.DT_F32, W.DT_BF16, W.DT_F32]
NUMELS = [1000, 777, 4096 + 37]
SEED, K, EPS = W.step_seed(3), 11, 1e-3


def initial_params():
    rng = np.random.default_rng(17)
    return [W.random_storage(rng, n, dt) for n, dt in zip(NUMELS, DTS)]


def coefficients_a():
    rng = np.random.default_rng(18)
    return [(10.0 ** rng.uniform(-2, 2, n)).astype(np.float32) for n in NUMELS]


def as_f32(t, dt):
    return t if dt == W.DT_F32 else oracle.bf16_to_f32(t)


def loss(tensors, a):
    """f = 1/2 sum_i a_i theta_i^2 over all tensors (oracle's quadratic loss)."""
    return float(sum(oracle.quadratic_loss(as_f32(t, dt), ai) for t, dt, ai in zip(tensors, DTS, a)))


def rows_pair(theta, a, probes):
    """Out-of-place: theta +- eps z_k on copies, theta untouched."""
    l0 = loss(theta, a)
    out = []
    for k in probes:
        plus, minus = [t.copy() for t in theta], [t.copy() for t in theta]
        oracle.perturb(plus, DTS, SEED, k, EPS)
        oracle.perturb(minus, DTS, SEED, k, -EPS)
        out.append((loss(plus, a), loss(minus, a), l0))
    return np.array(out, dtype=np.float64).reshape(-1, 3)


def rows_inplace(theta, a, probes):
    """Algorithm 1's in-place sequence on theta (left with its drift)."""
    l0 = loss(theta, a)
    out = []
    for k in probes:
        oracle.perturb(theta, DTS, SEED, k, EPS)
        lp = loss(theta, a)
        oracle.perturb(theta, DTS, SEED, k, -2 * EPS)
        lm = loss(theta, a)
        oracle.perturb(theta, DTS, SEED, k, EPS)
        out.append((lp, lm, l0))
    return np.array(out, dtype=np.float64).reshape(-1, 3)


def finish(theta, table):
    rc, c, _, _ = oracle.precondition(table, EPS)
    assert rc == oracle.OK
    oracle.update(theta, DTS, SEED, c, EPS)


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_worker(rank, world, port, schedule, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        theta, a = initial_params(), coefficients_a()
        mine = R.probes_of_rank(K, rank, world)
        own = rows_pair(theta, a, mine) if schedule == "pair" else rows_inplace(theta, a, mine)
        table = R.all_gather_losses(torch.from_numpy(own), K).numpy()
        finish(theta, table)
        if schedule == "inplace":
            R.broadcast_params([torch.from_numpy(t.view(np.uint8)) for t in theta], src=0)   # into the numpy storage
        out.put((rank, table, [t.copy() for t in theta]))
    finally:
        dist.destroy_process_group()


def run_ranks(world, schedule):
    port = free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=rank_worker, args=(r, world, port, schedule, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=300) for _ in range(world)), key=lambda x: x[0])
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    return res


def assert_same_storage(a, b, what):
    for i, (x, y) in enumerate(zip(a, b)):
        view = np.uint32 if x.dtype == np.float32 else np.uint16
        np.testing.assert_array_equal(x.view(view), y.view(view), err_msg=f"{what}: tensor {i}")


@pytest.mark.parametrize("world", [2, 3])
def test_gloo_pair_schedule_replicas_stay_identical(world):
    """Pair schedule: every rank gets the one-process table bit for bit and
    ends with the one-process parameters, with no parameter broadcast."""
    theta, a = initial_params(), coefficients_a()
    want_table = rows_pair(theta, a, range(K))
    finish(theta, want_table)
    for rank, table, th in run_ranks(world, "pair"):
        np.testing.assert_array_equal(table, want_table, err_msg=f"rank {rank} table")
        assert_same_storage(th, theta, f"rank {rank} parameters")


def test_gloo_inplace_schedule_broadcasts_rank0():
    """In-place schedule: each rank's restores leave its own drift, so after
    the update every rank holds rank 0's parameters, which are the oracle's
    in-place sequence over rank 0's probes followed by the update with the
    full table."""
    world = 2
    res = run_ranks(world, "inplace")
    theta, a = initial_params(), coefficients_a()
    parts = [rows_inplace([t.copy() for t in initial_params()], a, R.probes_of_rank(K, r, world))
             for r in range(world)]
    table = R.assemble_losses([torch.from_numpy(p) for p in parts], K, world).numpy()
    rows_inplace(theta, a, R.probes_of_rank(K, 0, world))
    finish(theta, table)
    other = initial_params()                # rank 1 without the broadcast: its own drift
    rows_inplace(other, a, R.probes_of_rank(K, 1, world))
    finish(other, table)
    assert any(not np.array_equal(x, y) for x, y in zip(theta, other)), "no drift: the broadcast is untested"
    for rank, tab, th in res:
        np.testing.assert_array_equal(tab, table, err_msg=f"rank {rank} table")
        assert_same_storage(th, theta, f"rank {rank} parameters")


# ------------------------------------------------------------------- the GPU
def gpu_setup(seed=5, n=(1 << 16) + 37):
    from paper_2609_38095_gb300 import build as zo_build
    from paper_2609_38095_gb300 import zo
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()
    rng = np.random.default_rng(seed)
    theta_h = W.random_storage(rng, n, W.DT_F32)
    a_h = (10.0 ** rng.uniform(-2, 2, n)).astype(np.float32)
    theta = torch.from_numpy(theta_h.copy()).cuda()
    a = torch.from_numpy(a_h).cuda()
    ws = torch.empty(zo.quadratic_loss_workspace_size(n), dtype=torch.uint8, device="cuda")

    def loss_into(tensors, out):
        zo.quadratic_loss(tensors[0], a, out=out, workspace=ws)

    return zo, theta_h, theta, loss_into


@pytest.mark.gpu
@pytest.mark.parametrize("schedule", ["pair", "inplace"])
def test_gpu_one_replica_step_matches_the_plain_schedule(schedule):
    """replicas.step without a process group is the single-GPU step: the
    same table and bit-identical parameters as the same calls made by hand."""
    zo, _, theta, loss_into = gpu_setup()
    Kg, eps, seed = 12, 1e-3, W.step_seed(9)
    ref = theta.clone()
    plus, minus = [torch.empty_like(theta)], [torch.empty_like(theta)]
    table, c, st = R.step([theta], seed, Kg, eps, loss_into, schedule=schedule, plus=plus, minus=minus)
    # by hand
    rows = torch.empty(Kg, 3, dtype=torch.float64, device="cuda")
    loss_into([ref], rows[0, 2:3])
    rows[:, 2] = rows[0, 2]
    if schedule == "pair":
        for k in range(Kg):
            zo.perturb_pair([ref], plus, minus, seed, k, eps)
            loss_into(plus, rows[k, 0:1])
            loss_into(minus, rows[k, 1:2])
        pre = None
    else:
        zo.perturb([ref], seed, 0, eps)
        for k in range(Kg):
            loss_into([ref], rows[k, 0:1])
            zo.perturb([ref], seed, k, -2 * eps)
            loss_into([ref], rows[k, 1:2])
            if k + 1 < Kg:
                zo.perturb2([ref], seed, k, eps, k + 1, eps)
        pre = (Kg - 1, eps)
    c2, st2 = zo.precondition(rows, eps)
    zo.update([ref], seed, c2, eps, status=st2, pre=pre)
    assert torch.equal(table, rows)
    assert torch.equal(c, c2)
    assert int(st.item()) == zo.ZO_OK
    assert torch.equal(theta.view(torch.int32), ref.view(torch.int32))


@pytest.mark.gpu
def test_gpu_three_replicas_pair_schedule():
    """Three replicas on one device, one after the other: each evaluates its
    probes (k = r mod 3) with the pair schedule; the assembled table equals
    the one-replica table and every replica ends bit-identical to the
    one-replica step -- with no parameter broadcast."""
    zo, theta_h, theta, loss_into = gpu_setup(seed=6)
    Kg, eps, seed, world = 14, 1e-3, W.step_seed(10), 3
    reps = [theta.clone() for _ in range(world)]
    plus, minus = [torch.empty_like(theta)], [torch.empty_like(theta)]
    l0 = torch.empty(1, dtype=torch.float64, device="cuda")
    parts = []
    for r in range(world):
        loss_into([reps[r]], l0)
        parts.append(R.pair_probe_losses([reps[r]], plus, minus, seed, Kg, eps, r, world, loss_into, l0))
    table = R.assemble_losses(parts, Kg, world)
    for r in range(world):
        assert torch.equal(reps[r].view(torch.int32), theta.view(torch.int32))   # probes left theta alone
        R.finish_step([reps[r]], table, seed, eps)
    one = theta.clone()
    table1, _, _ = R.step([one], seed, Kg, eps, loss_into, schedule="pair", plus=plus, minus=minus)
    assert torch.equal(table, table1)
    for r in range(world):
        assert torch.equal(reps[r].view(torch.int32), one.view(torch.int32)), f"replica {r}"
    # and the oracle's update of the unperturbed theta with that table
    rc, c_o, _, _ = oracle.precondition(table.cpu().numpy(), eps)
    assert rc == oracle.OK
    host = [theta_h.copy()]
    oracle.update(host, [W.DT_F32], seed, c_o, eps)
    assert_update_close(storage_bits(one), storage_bits(host[0]), W.DT_F32, c_o, eps, context="three replicas")


@pytest.mark.gpu
def test_gpu_three_replicas_inplace_schedule():
    """In-place schedule on three simulated replicas: each replica's
    parameters after its probes and the update are the oracle's in-place
    sequence over that replica's probes followed by the update with the
    full table (restores bit for bit, the update within its bound). Which
    replica's parameters the others then take is the broadcast's business
    (tested on gloo ranks above)."""
    zo, theta_h, theta, loss_into = gpu_setup(seed=7)
    Kg, eps, seed, world = 10, 1e-3, W.step_seed(11), 3
    reps = [theta.clone() for _ in range(world)]
    l0 = torch.empty(1, dtype=torch.float64, device="cuda")
    parts, pend = [], []
    for r in range(world):
        loss_into([reps[r]], l0)
        rows, pending = R.inplace_probe_losses([reps[r]], seed, Kg, eps, r, world, loss_into, l0)
        parts.append(rows)
        pend.append(pending)
    table = R.assemble_losses(parts, Kg, world)
    for r in range(world):
        c, _ = R.finish_step([reps[r]], table, seed, eps, pending=pend[r])
        host = [theta_h.copy()]
        for k in R.probes_of_rank(Kg, r, world):
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
        oracle.update(host, [W.DT_F32], seed, c.cpu().numpy(), eps)
        assert_update_close(storage_bits(reps[r]), storage_bits(host[0]), W.DT_F32, c.cpu().numpy(), eps,
                            context=f"replica {r}")
