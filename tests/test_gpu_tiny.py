"""The small workload (d = 2^20 fp32, quadratic loss, K = 8, eps = 1e-3,
lr = 1e-2) run free for ten full steps on the device (paper_2609_38095_gb300
.quadratic, every loss computed on the device) and by the oracle on its own:
the two trajectories share only their start. (The lockstep comparison, each
step started from the device's weights, is test_tiny_workload_lockstep.)

At lr = 1e-2 the workload is unstable -- its loss grows about a hundredfold
per step -- and so does any difference between two trajectories: the fused
update's fp32 sum and the oracle's exact sum differ by an fp32 rounding in a
few weights, and that difference grows about 200-fold per step (emulating the
kernel's summation order on the CPU gives 3e-8, 2e-7, 3e-5, 6e-3 at steps 1-4,
whatever the implementation). So the 1e-5 bar for free-running losses holds
for the steps before the loss has grown 10^5-fold at lr = 1e-2, and for all
ten steps at lr = 1e-5, where the workload is stable."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300.quadratic import QuadraticStep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def oracle_trajectory(steps, K, eps, lr):
    """Algorithm 1 on the oracle: per step the clean loss, per probe +eps,
    loss, -2 eps, loss, +eps, the preconditioner and the fused update."""
    host = [W.tiny_theta()]
    a = W.tiny_curvatures()
    tables = []
    for s in range(steps):
        seed = W.step_seed(s)
        l0 = oracle.quadratic_loss(host[0], a)
        rows = []
        for k in range(K):
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            lp = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
            lm = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            rows.append([lp, lm, l0])
        rows = np.array(rows)
        rc, c, _, _ = oracle.precondition(rows, eps)
        assert rc == oracle.OK
        oracle.update(host, [W.DT_F32], seed, c, lr)
        tables.append(rows)
    return tables, host[0]


def device_trajectory(steps, K, eps, lr, schedule):
    theta = torch.from_numpy(W.tiny_theta()).cuda()
    a = torch.from_numpy(W.tiny_curvatures()).cuda()
    q = QuadraticStep(theta, a, K, eps, lr, schedule=schedule)
    tables = []
    for s in range(steps):
        q.step(W.step_seed(s))
        tables.append(q.losses.cpu().numpy().copy())
        assert int(q.status.item()) == 0
    return tables, theta.cpu().numpy()


def rel_diff(got, want):
    return [float(np.max(np.abs(g - w) / np.abs(w))) for g, w in zip(got, want)]


@pytest.mark.parametrize("schedule", ["fused", "onepass"])
def test_free_running_trajectory_matches_the_oracle(schedule):
    ps = W.TINY
    K, eps, lr = ps.K, ps.eps, W.TINY_LR
    want, _ = oracle_trajectory(W.TINY_STEPS, K, eps, lr)
    got, _ = device_trajectory(W.TINY_STEPS, K, eps, lr, schedule)
    rel = rel_diff(got, want)
    growth = [w[0, 2] / want[0][0, 2] for w in want]
    print(f"free-running small workload ({schedule}), lr = 1e-2: relative loss drift per step",
          " ".join(f"{r:.1e}" for r in rel), "; loss growth", " ".join(f"{g:.1e}" for g in growth))
    stable = [s for s, g in enumerate(growth) if g < 1e5]
    assert len(stable) >= 3
    for s in stable:
        np.testing.assert_allclose(got[s], want[s], rtol=1e-5, err_msg=f"step {s}")
    # both runs blow up alike: every loss finite and growing
    assert all(np.all(np.isfinite(g)) for g in got)
    assert got[-1][0, 2] > got[0][0, 2] and want[-1][0, 2] > want[0][0, 2]


@pytest.mark.parametrize("schedule", ["fused", "onepass"])
def test_free_running_trajectory_at_a_stable_step_size(schedule):
    ps = W.TINY
    K, eps, lr = ps.K, ps.eps, 1e-5
    want, _ = oracle_trajectory(W.TINY_STEPS, K, eps, lr)
    got, _ = device_trajectory(W.TINY_STEPS, K, eps, lr, schedule)
    for s, (g, w) in enumerate(zip(got, want)):
        np.testing.assert_allclose(g, w, rtol=1e-5, err_msg=f"step {s}")
    print(f"free-running small workload ({schedule}), lr = 1e-5: relative loss drift per step",
          " ".join(f"{r:.1e}" for r in rel_diff(got, want)))


def test_fused_and_algorithm1_schedules_give_the_same_trajectory():
    ps = W.TINY
    a, th_a = device_trajectory(3, ps.K, ps.eps, W.TINY_LR, "fused")
    b, th_b = device_trajectory(3, ps.K, ps.eps, W.TINY_LR, "alg1")
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    np.testing.assert_array_equal(th_a.view(np.uint32), th_b.view(np.uint32))


def test_restore_exactness_and_drift_on_the_small_workload():
    """Algorithm 1's +eps, -2 eps, +eps per probe on the device, probe by
    probe over the small workload's K probes: bit-exact with the oracle after
    every probe, and the fraction of weights restored exactly and the largest
    drift (in ulps of |theta| + 2 eps, three correctly rounded adds allow 1.5)
    reported. Measured: 71.3 % exact after probe 0, 87.8-88.8 % after the
    others, drift at most 1 ulp; 72.2 % of the weights equal their start after
    all eight probes."""
    from paper_2609_38095_gb300 import zo
    ps = W.TINY
    eps, K, seed = ps.eps, ps.K, W.step_seed(0)
    start = W.tiny_theta()
    theta = torch.from_numpy(start).cuda()
    plist = zo.ParamList([theta])
    host = [start.copy()]
    exact = []
    for k in range(K):
        before = host[0].copy()
        for s in (eps, -2 * eps, eps):
            zo.perturb(plist, seed, k, s)
            oracle.perturb(host, [W.DT_F32], seed, k, s)
        got = theta.cpu().numpy()
        np.testing.assert_array_equal(got.view(np.uint32), host[0].view(np.uint32), err_msg=f"probe {k}")
        drift = np.abs(got.astype(np.float64) - before)
        unit = np.spacing((np.abs(before) + 2 * eps).astype(np.float32)).astype(np.float64)
        exact.append(float(np.mean(drift == 0)))
        assert np.max(drift / unit) <= 1.5, f"probe {k}"
    total = float(np.mean(theta.cpu().numpy() == start))
    print("restore after each probe: exactly restored", " ".join(f"{e:.4f}" for e in exact),
          f"; equal to the start after {K} probes: {total:.4f}")
    assert min(exact) > 0.5 and total > 0.5


def test_step_rejects_mismatched_inputs():
    theta = torch.zeros(16, dtype=torch.float32, device="cuda")
    with pytest.raises(ValueError):
        QuadraticStep(theta, torch.zeros(8, dtype=torch.float32, device="cuda"), 8, 1e-3, 1e-2)
    with pytest.raises(ValueError):
        QuadraticStep(theta, torch.zeros(16, dtype=torch.float64, device="cuda"), 8, 1e-3, 1e-2)
    with pytest.raises(ValueError):
        QuadraticStep(theta, torch.zeros(16, dtype=torch.float32, device="cuda"), 8, 1e-3, 1e-2, schedule="x")
