"""The stiff-paraboloid sweep (Sec. 5.3): the problem's construction (CPU),
its step against the oracle in lockstep, and a short sweep (GPU)."""
import numpy as np
import pytest
import torch

import oracle
import paraboloid_sweep as ps
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

from gpu_helpers import assert_update_close, storage_bits


@pytest.mark.parametrize("k", [1.0, 37.0, 1000.0])
def test_problem_is_a_rotated_diagonal(k):
    """M = R^T diag(k, 1, ..., 1) R with R orthonormal: eigenvalues {k, 1, ...},
    J(x) = |D^(1/2) R x|^2."""
    p = ps.Paraboloid(10, k, seed=3, device="cpu")
    R = p.R.numpy()
    np.testing.assert_allclose(R.T @ R, np.eye(10), atol=1e-12)
    ev = np.sort(np.linalg.eigvalsh(p.M.numpy()))
    np.testing.assert_allclose(ev, np.sort([k] + [1.0] * 9), rtol=1e-10)
    x = p.x0
    out = torch.empty((), dtype=torch.float64)
    p.loss_into(x, out)
    d = np.ones(10)
    d[0] = k
    want = float(np.sum(d * (R @ x.double().numpy()) ** 2))
    assert float(out) == pytest.approx(want, rel=1e-12)


def test_step_seeds_and_grid_defaults():
    a = ps.parse_args([])
    assert [float(v) for v in a.kappas.split(",")] == [1, 5, 10, 50, 100, 500, 1000]
    assert a.seeds == 10 and ps.SOLVERS == {"1SPSA": 0.0, "1.5-SPSA": 0.1}


@pytest.mark.gpu
def test_paraboloid_steps_match_the_oracle():
    """Five steps of 1.5-SPSA on the paraboloid: each step starts the oracle
    from the GPU's weights; losses, coefficients and the updated weights
    agree (perturbations bit for bit, losses up to the fp64 summation order,
    the update within its tolerance)."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()
    dev = torch.device("cuda")
    K, eps, alpha = 8, 0.03, 0.1
    p = ps.Paraboloid(10, 100.0, seed=5, device=dev)
    M = p.M.cpu().numpy()
    x = p.x0.clone()
    plist = zo.ParamList([x])
    losses = torch.empty(K, 3, dtype=torch.float64, device=dev)
    c = torch.empty(K, dtype=torch.float64, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)

    def J(v):
        vd = v.astype(np.float64)
        return float(vd @ (M @ vd))

    for s in range(5):
        seed = ps.STEP_SEED_BASE + s
        host = [x.cpu().numpy().copy()]
        ps.step(p, plist, x, seed, K, eps, alpha, losses, c, st)
        rows = []
        l0 = J(host[0])
        for k in range(K):
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            lp = J(host[0])
            oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
            lm = J(host[0])
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            rows.append([lp, lm, l0])
        Lg = losses.cpu().numpy()
        np.testing.assert_allclose(Lg, np.array(rows), rtol=1e-12)
        assert int(st.item()) == zo.ZO_OK
        rc, c_o, _, _ = oracle.precondition(Lg, eps, alpha=alpha, lambda_reg=1.0)
        assert rc == oracle.OK
        np.testing.assert_allclose(c.cpu().numpy(), c_o, rtol=1e-12)
        oracle.update(host, [W.DT_F32], seed, c.cpu().numpy(), eps)
        assert_update_close(storage_bits(x), storage_bits(host[0]), W.DT_F32, c.cpu().numpy(), eps,
                            context=f"step {s}")


@pytest.mark.gpu
def test_short_sweep_runs():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    rows = ps.sweep(ps.parse_args(["--kappas", "10", "--seeds", "2", "--search-seeds", "1",
                                   "--eps-grid", "0.1,0.03", "--max-steps", "400"]))
    assert len(rows) == 1
    for name in ps.SOLVERS:
        r = rows[0][name]
        assert r["eps"] in (0.1, 0.03) and len(r["steps"]) == 2
