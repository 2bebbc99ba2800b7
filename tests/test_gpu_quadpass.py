"""zo_perturb_quadratic_loss: one forward point of the small workload in one
launch -- up to two perturbations of theta and the quadratic loss of the
result -- against the oracle's perturbation (bit for bit) and its fp64 loss
(within 1e-12 relative), on sizes that span several CTAs and a ragged last
block, both packings, views off the 16-byte grid, special values, repeated
calls on one workspace, and the small workload's step in lockstep."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo
from paper_2609_38095_gb300.quadratic import QuadraticStep

from gpu_helpers import assert_update_close, storage_bits

pytestmark = pytest.mark.gpu

OPS = {"none": (), "one": ((3, 1e-3),), "same-group": ((3, 1e-3), (4, -2e-3)),
       "two-groups": ((7, 1e-3), (8, 1e-3))}


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def oracle_pass(theta, a, seed, ops):
    host = [theta.copy()]
    for k, s in ops:
        oracle.perturb(host, [W.DT_F32], seed, k, s)
    return host[0], oracle.quadratic_loss(host[0], a)


def on_device(x, offset):
    """x on the device, `offset` elements into its own allocation."""
    buf = torch.zeros(x.size + offset, dtype=torch.float32, device="cuda")
    v = buf[offset:]
    v.copy_(torch.from_numpy(x))
    return v


@pytest.mark.parametrize("n", [0, 1, 15, 16, 17, 4099, 65536 + 5, 1 << 20, 3_000_001])
@pytest.mark.parametrize("ops", list(OPS))
def test_quadpass_parity(n, ops):
    rng = np.random.default_rng(n + len(ops))
    th = W.random_storage(rng, n, W.DT_F32)
    a = (10.0 ** rng.uniform(-2, 2, n)).astype(np.float32)
    seed = W.step_seed(n)
    theta, ad = on_device(th, 0), on_device(a, 0)
    out = torch.full((1,), -1.0, dtype=torch.float64, device="cuda")
    zo.perturb_quadratic_loss(theta, ad, seed, OPS[ops], out=out)
    want_th, want_l = oracle_pass(th, a, seed, OPS[ops])
    np.testing.assert_array_equal(theta.cpu().numpy().view(np.uint32), want_th.view(np.uint32))
    got = float(out.item())
    assert got == want_l if want_l == 0 else abs(got - want_l) <= 1e-12 * abs(want_l), (got, want_l)


@pytest.mark.parametrize("offset_theta,offset_a", [(1, 0), (0, 3), (2, 1)])
@pytest.mark.parametrize("packing", [1, 8])
def test_quadpass_views_and_packings(offset_theta, offset_a, packing):
    """Views off the 16-byte grid take the scalar loads; the packing named
    in the call (or the process default) decides the probes, as for a
    parameter list."""
    n = 100003
    rng = np.random.default_rng(packing * 10 + offset_theta)
    th = W.random_storage(rng, n, W.DT_F32)
    a = (10.0 ** rng.uniform(-2, 2, n)).astype(np.float32)
    seed = W.step_seed(7)
    for named in (True, False):
        theta, ad = on_device(th, offset_theta), on_device(a, offset_a)
        out = torch.empty(1, dtype=torch.float64, device="cuda")
        if named:
            zo.perturb_quadratic_loss(theta, ad, seed, OPS["two-groups"], out=out, packing=packing)
        else:
            with zo.packing(packing):
                zo.perturb_quadratic_loss(theta, ad, seed, OPS["two-groups"], out=out)
        with oracle.packing(packing):
            want_th, want_l = oracle_pass(th, a, seed, OPS["two-groups"])
        np.testing.assert_array_equal(theta.cpu().numpy().view(np.uint32), want_th.view(np.uint32))
        assert abs(float(out.item()) - want_l) <= 1e-12 * abs(want_l)


def test_quadpass_out_copies_and_repeated_calls():
    """The loss goes to out[j * stride], j < copies, and nothing else; one
    workspace serves call after call (its counter is left at zero)."""
    n, K = 50001, 8
    rng = np.random.default_rng(5)
    th = W.random_storage(rng, n, W.DT_F32)
    a = (10.0 ** rng.uniform(-2, 2, n)).astype(np.float32)
    theta, ad = on_device(th, 0), on_device(a, 0)
    q = zo.QuadraticPass(theta, ad)
    table = torch.full((K, 3), -7.0, dtype=torch.float64, device="cuda")
    seed = W.step_seed(3)
    q(seed, (), q.out_address(table) + 16, copies=K, stride=3)          # the third column
    want0 = oracle.quadratic_loss(th, a)
    t = table.cpu().numpy()
    assert np.all(t[:, :2] == -7.0)
    np.testing.assert_allclose(t[:, 2], want0, rtol=1e-12)
    host = th.copy()
    for k in range(K):                                                    # then one cell per call
        q(seed, ((k, 1e-3),), q.out_address(table) + 24 * k)
        host, want = oracle_pass(host, a, seed, ((k, 1e-3),))
        assert abs(table[k, 0].item() - want) <= 1e-12 * abs(want), k
    np.testing.assert_array_equal(theta.cpu().numpy().view(np.uint32), host.view(np.uint32))


def test_quadpass_special_values():
    """Infinities, NaN, zeros, subnormals and weights whose square leaves
    fp32's range (their terms go to fp64): NaN where the oracle has NaN, an
    infinite loss where it has one, else within 1e-12 relative."""
    base = np.array([0.0, -0.0, 1e-30, -1e-30, 1e-40, 3e-39, 1e19, -1e19, 1e30, 3.3e38, 1.0, -2.5, 0.02],
                    dtype=np.float32)
    cases = {
        "finite": (base, np.full(base.size, 3.0, dtype=np.float32)),
        "zero curvature": (base, np.where(np.arange(base.size) % 2 == 0, 0.0, 5.0).astype(np.float32)),
        "tiny only": (np.array([1e-30, 2e-25, -3e-28, 1e-38], dtype=np.float32), np.ones(4, dtype=np.float32)),
        "with inf": (np.append(base, np.float32(np.inf)), np.ones(base.size + 1, dtype=np.float32)),
        "inf times 0": (np.append(base, np.float32(np.inf)), np.zeros(base.size + 1, dtype=np.float32)),
        "with nan": (np.append(base, np.float32(np.nan)), np.ones(base.size + 1, dtype=np.float32)),
    }
    for name, (th, a) in cases.items():
        for ops in (OPS["none"], OPS["one"]):
            theta, ad = on_device(th, 0), on_device(a, 0)
            out = torch.empty(1, dtype=torch.float64, device="cuda")
            zo.perturb_quadratic_loss(theta, ad, W.step_seed(1), ops, out=out)
            want_th, want = oracle_pass(th, a, W.step_seed(1), ops)
            np.testing.assert_array_equal(theta.cpu().numpy().view(np.uint32), want_th.view(np.uint32))
            got = float(out.item())
            if np.isnan(want) or np.isinf(want):
                assert (np.isnan(got) and np.isnan(want)) or got == want, (name, got, want)
            else:
                assert abs(got - want) <= 1e-12 * abs(want) or got == want, (name, got, want)


def test_quadpass_argument_errors():
    theta = torch.zeros(64, dtype=torch.float32, device="cuda")
    a = torch.ones(64, dtype=torch.float32, device="cuda")
    out = torch.empty(1, dtype=torch.float64, device="cuda")
    q = zo.QuadraticPass(theta, a)
    L = zo._lib()
    ws = torch.zeros(zo.perturb_quadratic_loss_workspace_size(64), dtype=torch.uint8, device="cuda")
    import ctypes
    args = (ctypes.c_void_p(theta.data_ptr()), ctypes.c_void_p(a.data_ptr()), 64, 1, 0)
    tail = (ctypes.c_void_p(ws.data_ptr()), ws.numel(), None)
    o = ctypes.c_void_p(out.data_ptr())
    assert L.zo_perturb_quadratic_loss(*args, 3, 0, 1e-3, 0, 0.0, o, 1, 1, *tail) == zo.ZO_ERR_ARG   # nops
    assert L.zo_perturb_quadratic_loss(*args, 1, 0, float("inf"), 0, 0.0, o, 1, 1, *tail) == zo.ZO_ERR_ARG
    assert L.zo_perturb_quadratic_loss(*args, 1, 0, 1e-3, 0, 0.0, o, 0, 1, *tail) == zo.ZO_ERR_ARG   # copies
    assert L.zo_perturb_quadratic_loss(*args, 1, 0, 1e-3, 0, 0.0, None, 1, 1, *tail) == zo.ZO_ERR_ARG
    bad_pack = (ctypes.c_void_p(theta.data_ptr()), ctypes.c_void_p(a.data_ptr()), 64, 1, 2)
    assert L.zo_perturb_quadratic_loss(*bad_pack, 1, 0, 1e-3, 0, 0.0, o, 1, 1, *tail) == zo.ZO_ERR_ARG
    small = (ctypes.c_void_p(ws.data_ptr()), 8, None)
    assert L.zo_perturb_quadratic_loss(*args, 1, 0, 1e-3, 0, 0.0, o, 1, 1, *small) == zo.ZO_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.all(theta == 0)                                        # nothing was enqueued
    with pytest.raises(ValueError):
        q(1, ((0, 1e-3), (1, 1e-3), (2, 1e-3)), q.out_address(out))
    with pytest.raises(ValueError):
        zo.QuadraticPass(theta, torch.ones(63, dtype=torch.float32, device="cuda"))


def test_tiny_workload_onepass_lockstep():
    """Ten full steps of the small workload with the onepass schedule
    (QuadraticStep, every forward point one launch). Each step starts the
    oracle from the device's weights: the losses within 1e-12, the
    preconditioner on the device's losses within 1e-12, the update within
    the derived bound."""
    ps = W.TINY
    theta = torch.from_numpy(W.tiny_theta()).cuda()
    a = W.tiny_curvatures()
    q = QuadraticStep(theta, torch.from_numpy(a).cuda(), ps.K, ps.eps, W.TINY_LR, schedule="onepass")
    K, eps, lr = ps.K, ps.eps, W.TINY_LR
    for step in range(W.TINY_STEPS):
        seed = W.step_seed(step)
        host = [theta.cpu().numpy().copy()]
        q.step(seed)
        rows = []
        l0 = oracle.quadratic_loss(host[0], a)
        for k in range(K):
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            lp = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
            lm = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            rows.append([lp, lm, l0])
        Lg = q.losses.cpu().numpy()
        assert int(q.status.item()) == zo.ZO_OK
        np.testing.assert_allclose(Lg, np.array(rows), rtol=1e-12, err_msg=f"step {step}")
        cg = q.c.cpu().numpy()
        rc, c_same, _, _ = oracle.precondition(Lg, eps)
        assert rc == oracle.OK
        np.testing.assert_allclose(cg, c_same, rtol=1e-12)
        oracle.update(host, [W.DT_F32], seed, cg, lr)
        assert_update_close(storage_bits(theta), storage_bits(host[0]), W.DT_F32, cg, lr, context=f"step {step}")


def test_tiny_onepass_step_replayed_from_a_cuda_graph():
    """The onepass step only enqueues work (its workspace counter is left at
    zero by every launch), so a captured step replays correctly: two replays
    from the same start give the eager step's losses, coefficients and
    weights bit for bit."""
    ps = W.TINY
    start = W.tiny_theta()
    a = torch.from_numpy(W.tiny_curvatures()).cuda()
    theta = torch.from_numpy(start.copy()).cuda()
    q = QuadraticStep(theta, a, ps.K, ps.eps, W.TINY_LR, schedule="onepass")
    q.step(W.step_seed(5))
    torch.cuda.synchronize()
    want = (q.losses.clone(), q.c.clone(), theta.clone())
    theta.copy_(torch.from_numpy(start))
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            q.step(W.step_seed(5))
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(2):
        theta.copy_(torch.from_numpy(start))
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(q.losses, want[0]) and torch.equal(q.c, want[1])
        assert torch.equal(theta.view(torch.int32), want[2].view(torch.int32))
