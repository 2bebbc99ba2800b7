"""Pins for the oracle's perturb, preconditioner, update and quadratic loss.

Each check rests on something other than the oracle's own formula: numpy's
fp32 arithmetic and library casts (brute force), exact-arithmetic identities
(restore on an exact grid, the quadratic closed forms of the FD-bias lemma in
the appendix), a value the paper prints (Sec. 6), the alpha special cases of
Sec. 4.1, and error bounds of fp32 summation.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def to_f32(raw, dtype):
    if dtype == W.DT_F32:
        return raw.astype(np.float32)
    if dtype == W.DT_F16:
        return raw.view(np.float16).astype(np.float32)
    return (raw.astype(np.uint32) << 16).view(np.float32)


def from_f32(x, dtype):
    """Round fp32 values to storage with numpy / torch casts (independent)."""
    x = np.asarray(x, dtype=np.float32)
    if dtype == W.DT_F32:
        return x
    if dtype == W.DT_F16:
        return x.astype(np.float16).view(np.uint16)
    return torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def from_f64(x, dtype):
    """One rounding from double to storage, via torch casts (independent)."""
    t = torch.from_numpy(np.asarray(x, dtype=np.float64))
    if dtype == W.DT_F32:
        return t.to(torch.float32).numpy()
    if dtype == W.DT_F16:
        return t.to(torch.float16).view(torch.int16).numpy().view(np.uint16)
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def ulp_f32(x):
    return np.spacing(np.abs(np.asarray(x, dtype=np.float32))).astype(np.float64)


def make_tensors(numels, dtypes, seed=0):
    rng = np.random.default_rng(seed)
    return [W.random_storage(rng, n, dt) for n, dt in zip(numels, dtypes)]


def signs_for(seed, k, numels):
    """z_k for each tensor via the virtual index (probe generator pinned in
    test_oracle_probe.py)."""
    S = oracle.virtual_offsets(numels)
    return [oracle.probe_signs(seed, k, int(s), int(n)).astype(np.float32) for s, n in zip(S, numels)]


NUMELS = [1, 17, 64, 1000, 4099, 33]
DTYPES = [W.DT_F32, W.DT_BF16, W.DT_F16, W.DT_BF16, W.DT_F32, W.DT_F16]


# ---------------------------------------------------------------- perturb
@pytest.mark.parametrize("scale", [1e-3, -2e-3, 0.5, 3e-8])
def test_perturb_brute_force(scale):
    seed, k = 0x15E5A0002, 9
    ts = make_tensors(NUMELS, DTYPES)
    before = [t.copy() for t in ts]
    oracle.perturb(ts, DTYPES, seed, k, scale)
    zs = signs_for(seed, k, NUMELS)
    for t, b, z, dt in zip(ts, before, zs, DTYPES):
        want = from_f32(to_f32(b, dt) + np.float32(scale) * z, dt)   # numpy fp32 add
        np.testing.assert_array_equal(t.view(np.uint32 if dt == W.DT_F32 else np.uint16),
                                      want.view(np.uint32 if dt == W.DT_F32 else np.uint16))


def test_perturb_restore_exact_on_grid():
    """theta on multiples of 2^-20 in (-0.25, 0.25), eps = 2^-10: every fp32
    add is exact, so +eps, -2 eps, +eps restores theta bit for bit."""
    rng = np.random.default_rng(5)
    theta = (rng.integers(-(2**18), 2**18, 50000) * 2.0 ** -20).astype(np.float32)
    t = [theta.copy()]
    eps = 2.0 ** -10
    seed, k = 0x15E5A0000, 3
    oracle.perturb(t, [W.DT_F32], seed, k, eps)
    assert np.any(t[0] != theta)
    oracle.perturb(t, [W.DT_F32], seed, k, -2 * eps)
    oracle.perturb(t, [W.DT_F32], seed, k, eps)
    np.testing.assert_array_equal(t[0], theta)


def test_perturb_restore_drift_bound_fp32():
    """Three correctly rounded adds: |theta'' - theta| <= 1.5 ulp(|theta| + 2 eps)."""
    theta = W.tiny_theta(1 << 16)
    t = [theta.copy()]
    eps = 1e-3
    seed, k = 0x15E5A0000, 0
    for s in (eps, -2 * eps, eps):
        oracle.perturb(t, [W.DT_F32], seed, k, s)
    drift = np.abs(t[0].astype(np.float64) - theta)
    bound = 1.5 * ulp_f32(np.abs(theta) + 2 * eps)
    assert np.all(drift <= bound)
    assert np.mean(drift == 0) > 0.5


# ----------------------------------------------------------- precondition
def test_precondition_worked_value_sec6():
    g = json.load(open(os.path.join(GOLDEN, "precondition_worked_value.json")))
    eps = 1e-3
    half = g["curvature"] * eps * eps / 2   # L+ = L- = half, L0 = 0 -> curvature 1e8
    rc, c, w, cv = oracle.precondition([[half, half, 0.0]], eps, alpha=g["alpha"], lambda_reg=g["lambda_reg"])
    assert rc == oracle.OK
    assert cv[0] == pytest.approx(g["curvature"], rel=1e-12)
    power = 1.0 / w[0]
    assert round(power, g["printed_power_digits"]) == g["printed_power"]
    assert round(power) == g["printed_downweight_vs_zero_curvature"]
    assert power == pytest.approx(10 ** 0.8, rel=1e-14)   # (1e8)^0.1 in exact arithmetic
    assert c[0] == 0.0                                     # L+ == L- -> no signal


def test_precondition_alpha_special_cases():
    g = json.load(open(os.path.join(GOLDEN, "alpha_special_cases.json")))
    rng = np.random.default_rng(2)
    eps = 1e-3
    L = np.column_stack([2.5 + rng.uniform(-0.05, 0.05, 64), 2.5 + rng.uniform(-0.05, 0.05, 64), np.full(64, 2.5)])
    L[0] = [2.5, 2.5, 2.5]          # zero curvature
    L[1] = [2.5 + 1e-7, 2.5, 2.5]   # |curvature| < 1
    for case in g["cases"]:
        rc, c, w, cv = oracle.precondition(L, eps, alpha=case["alpha"], lambda_reg=g["lambda_reg"])
        assert rc == oracle.OK
        if case["alpha"] == 0.0:
            np.testing.assert_array_equal(w, 1.0)
            # 1SPSA central difference (Sec. 2): (L+ - L-) / (2 eps)
            np.testing.assert_allclose(c, (L[:, 0] - L[:, 1]) / (2 * eps), rtol=1e-15)
        else:
            np.testing.assert_allclose(w, 1.0 / np.maximum(1.0, np.abs(cv)), rtol=1e-15)
            assert w[0] == 1.0 and w[1] == 1.0


def test_precondition_hand_example():
    """L+ = 3.04, L- = 2.98, L0 = 3.0, eps = 0.01: curvature = 0.02/1e-4 = 200,
    w = 1 / 200^0.1, c = w * 0.06 / 0.02 = 3 w; one-sided c = w * 0.04 / 0.01."""
    L = [[3.04, 2.98, 3.0]]
    rc, c, w, cv = oracle.precondition(L, 0.01)
    assert rc == oracle.OK
    assert cv[0] == pytest.approx(200.0, rel=1e-9)
    assert w[0] == pytest.approx(200.0 ** -0.1, rel=1e-9)
    assert c[0] == pytest.approx(3.0 * 200.0 ** -0.1, rel=1e-9)
    rc, c1, w1, _ = oracle.precondition(L, 0.01, one_sided=True)
    assert c1[0] == pytest.approx(4.0 * 200.0 ** -0.1, rel=1e-9)
    # lambda_reg floor: with lambda_reg = 3 > 200^0.1 = 1.698, w = 1/3
    rc, c2, w2, _ = oracle.precondition(L, 0.01, lambda_reg=3.0)
    assert w2[0] == pytest.approx(1.0 / 3.0, rel=1e-15)
    # negative curvature uses |curvature|
    rc, c3, w3, cv3 = oracle.precondition([[2.98, 2.96, 3.0]], 0.01)
    assert cv3[0] == pytest.approx(-600.0, rel=1e-9) and w3[0] == pytest.approx(600.0 ** -0.1, rel=1e-9)


@pytest.mark.parametrize("bad", [np.nan, np.inf, -np.inf])
@pytest.mark.parametrize("col", [0, 1, 2])
def test_precondition_nonfinite(bad, col):
    L = np.array([[2.5, 2.4, 2.45], [2.6, 2.3, 2.45]])
    L[1, col] = bad
    rc, c, w, cv = oracle.precondition(L, 1e-3)
    assert rc == oracle.ERR_NONFINITE
    assert np.all(np.isnan(c)) and np.all(np.isnan(w))   # nothing written


def test_precondition_curvature_overflow_is_nonfinite():
    rc, c, w, cv = oracle.precondition([[1e300, 1e300, -1e300]], 1e-300)
    assert rc == oracle.ERR_NONFINITE


def test_precondition_bad_args():
    assert oracle.precondition([[1, 1, 1]], 0.0)[0] == oracle.ERR_ARG
    assert oracle.precondition([[1, 1, 1]], 1e-3, alpha=1.5)[0] == oracle.ERR_ARG
    assert oracle.precondition([[1, 1, 1]], 1e-3, lambda_reg=0.0)[0] == oracle.ERR_ARG
    for bad_flags in (4, 8, -1):
        assert oracle.precondition([[1, 1, 1]], 1e-3, flags=bad_flags)[0] == oracle.ERR_ARG


# ------------------------------------------- relative curvature (Sec. 6 reading)
def triples_with_curvature(g, curv, eps):
    """(L+, L-, L0) rows with first difference g and curvature curv:
    L0 = 0, L+- = +-g eps + curv eps^2 / 2."""
    g, curv = np.asarray(g, float), np.asarray(curv, float)
    return np.column_stack([g * eps + curv * eps * eps / 2, -g * eps + curv * eps * eps / 2, np.zeros_like(g)])


def test_relative_curvature_alpha1_closed_form():
    """alpha = 1 and a negligible floor: w_k = m / |curv_k|, so sum_k 1/w_k = K
    and w_k |curv_k| is the same for every probe (= m, the mean |curvature|)."""
    eps = 1e-2
    curv = np.array([1.0, 1.0, 1.0, 5.0, -3.0, 0.5, 20.0, -7.5])
    g = np.linspace(-1, 1, len(curv))
    rc, c, w, cv = oracle.precondition(triples_with_curvature(g, curv, eps), eps, alpha=1.0, lambda_reg=1e-12,
                                       relative=True)
    assert rc == oracle.OK
    m = np.mean(np.abs(curv))
    np.testing.assert_allclose(cv, curv, rtol=1e-9)             # curv is still Eq. 3's curvature
    np.testing.assert_allclose(w * np.abs(cv), m, rtol=1e-9)
    assert np.sum(1.0 / w) == pytest.approx(len(curv), rel=1e-12)
    np.testing.assert_allclose(c, w * g, rtol=1e-9)              # central difference unchanged


def test_relative_curvature_equal_magnitudes():
    """Equal |curvature| in every probe: every ratio is +-1, so w = 1/max(lambda, 1)
    whatever alpha and the common magnitude (a plain sum instead of the mean would
    give ratios 1/K and w = K^alpha here)."""
    eps = 1e-3
    for mag in (1e-3, 1.0, 3e4):
        curv = mag * np.array([1, -1, 1, 1, -1, -1, 1, 1, 1, -1, 1, 1])
        for alpha in (0.1, 0.5, 1.0):
            rc, c, w, _ = oracle.precondition(triples_with_curvature(np.ones(12), curv, eps), eps, alpha=alpha,
                                              lambda_reg=1e-3, relative=True)
            assert rc == oracle.OK
            np.testing.assert_allclose(w, 1.0, rtol=1e-12)


def test_relative_curvature_scale_invariance():
    """Scaling every curvature by s leaves the relative weights unchanged, while
    the paper's absolute weights move by s^-alpha where the floor is inactive."""
    rng = np.random.default_rng(9)
    eps = 1e-3
    curv = rng.uniform(-2e4, 2e4, 64)
    g = rng.uniform(-50, 50, 64)
    _, _, w1, _ = oracle.precondition(triples_with_curvature(g, curv, eps), eps, relative=True)
    for s in (1e-3, 10.0, 1e3):
        _, _, ws, _ = oracle.precondition(triples_with_curvature(g, s * curv, eps), eps, relative=True)
        np.testing.assert_allclose(ws, w1, rtol=1e-6)
    _, _, a1, _ = oracle.precondition(triples_with_curvature(g, curv, eps), eps)
    _, _, a2, _ = oracle.precondition(triples_with_curvature(g, 1e3 * curv, eps), eps)
    big = np.abs(curv) > 10
    np.testing.assert_allclose(a2[big], a1[big] * 1e3 ** -0.1, rtol=1e-6)


def test_relative_curvature_degenerate_cases():
    eps = 1e-3
    # K = 1: the ratio is +-1
    rc, _, w, _ = oracle.precondition(triples_with_curvature([2.0], [-123.0], eps), eps, alpha=0.7,
                                      lambda_reg=1e-3, relative=True)
    assert rc == oracle.OK and w[0] == pytest.approx(1.0, rel=1e-12)
    # every curvature zero: m = 0, ratios 0, w = 1 / lambda_reg
    rc, c, w, _ = oracle.precondition([[2.0, 2.0, 2.0], [2.5, 1.5, 2.0]], eps, lambda_reg=0.5, relative=True)
    assert rc == oracle.OK
    np.testing.assert_array_equal(w, 2.0)
    assert c[1] == pytest.approx(2.0 * 1.0 / (2 * eps), rel=1e-12)
    # combined with the one-sided difference
    rc, c, w, _ = oracle.precondition([[3.04, 2.98, 3.0]], 0.01, alpha=1.0, lambda_reg=1e-9, relative=True,
                                      one_sided=True)
    assert w[0] == pytest.approx(1.0, rel=1e-12) and c[0] == pytest.approx(4.0, rel=1e-9)
    # a sum of |curvature| overflowing to infinity is non-finite
    big = 1.5e308 * 1e-6 / 2
    rc, c, _, _ = oracle.precondition([[big, big, 0.0], [big, big, 0.0]], 1e-3, relative=True)
    assert rc == oracle.ERR_NONFINITE and np.all(np.isnan(c))


def quad_setup(d=4096, seed=11):
    """Quadratic with theta on a 2^-20 grid and eps = 2^-10 so that the
    perturbed weights are exact; a_i log-uniform as in the small workload."""
    rng = np.random.default_rng(seed)
    theta = (rng.integers(-(2**14), 2**14, d) * 2.0 ** -20).astype(np.float32)
    a = (10.0 ** rng.uniform(-2, 2, d)).astype(np.float32)
    return theta, a


@pytest.mark.parametrize("k", [0, 1, 7, 8, 100])
def test_quadratic_closed_forms(k):
    """FD-bias lemma (appendix) with zero third derivative: for
    f = 1/2 sum a_i theta_i^2 and Rademacher z,
        (L+ - 2 L0 + L-) / eps^2 = z^T A z = sum_i a_i    (Eq. 3 is exact)
        (L+ - L-) / (2 eps)       = z^T A theta          (the SPSA numerator)."""
    theta, a = quad_setup()
    eps = 2.0 ** -10
    seed = 0x15E5A0005
    t = [theta.copy()]
    L0 = oracle.quadratic_loss(t[0], a)
    oracle.perturb(t, [W.DT_F32], seed, k, eps)
    Lp = oracle.quadratic_loss(t[0], a)
    oracle.perturb(t, [W.DT_F32], seed, k, -2 * eps)
    Lm = oracle.quadratic_loss(t[0], a)
    oracle.perturb(t, [W.DT_F32], seed, k, eps)
    np.testing.assert_array_equal(t[0], theta)
    rc, c, w, cv = oracle.precondition([[Lp, Lm, L0]], eps, alpha=0.0)
    assert rc == oracle.OK
    sum_a = math.fsum(a.astype(np.float64))
    assert cv[0] == pytest.approx(sum_a, rel=1e-9)
    z = oracle.probe_signs(seed, k, 0, theta.size).astype(np.float64)
    grad_dir = math.fsum(a.astype(np.float64) * z * theta.astype(np.float64))
    assert c[0] == pytest.approx(grad_dir, rel=1e-7, abs=1e-9 * sum_a)


# ----------------------------------------------------------------- update
def update_coeffs(c, lr):
    m = -(lr / len(c))
    return np.array([np.float32(m * ci) for ci in c], dtype=np.float32)


@pytest.mark.parametrize("K", [1, 3, 8, 13, 64])
def test_update_fp64_brute_force(K):
    seed = 0x15E5A0007
    rng = np.random.default_rng(K)
    c = rng.normal(0, 25, K)
    lr = 1e-3
    ts = make_tensors(NUMELS, DTYPES, seed=K)
    before = [t.copy() for t in ts]
    oracle.update(ts, DTYPES, seed, c, lr)
    a = update_coeffs(c, lr).astype(np.float64)
    zk = [signs_for(seed, k, NUMELS) for k in range(K)]
    for ti, (t, b, dt) in enumerate(zip(ts, before, DTYPES)):
        acc = np.zeros(b.size)
        for k in range(K):
            acc = acc + a[k] * zk[k][ti].astype(np.float64)
        want = from_f64(to_f32(b, dt).astype(np.float64) + acc, dt)
        np.testing.assert_array_equal(t, want)


def test_update_K1_equals_perturb_fp32():
    seed, c, lr = 0x15E5A0001, [3.7], 2e-3
    ts = make_tensors([5000], [W.DT_F32])
    t2 = [ts[0].copy()]
    oracle.update(ts, [W.DT_F32], seed, c, lr)
    oracle.perturb(t2, [W.DT_F32], seed, 0, float(update_coeffs(c, lr)[0]))
    np.testing.assert_array_equal(ts[0], t2[0])


def test_update_linearity_fp32():
    """update(c) then update(-c): two correctly rounded adds, so theta returns
    within 1/2 ulp(|theta| + sum|a|) + 1/2 ulp(theta)."""
    seed, lr = 0x15E5A0004, 1e-3
    c = np.random.default_rng(4).normal(0, 10, 16)
    theta = W.tiny_theta(8192)
    t = [theta.copy()]
    oracle.update(t, [W.DT_F32], seed, c, lr)
    assert np.any(t[0] != theta)
    oracle.update(t, [W.DT_F32], seed, -c, lr)
    S = np.abs(update_coeffs(c, lr).astype(np.float64)).sum()
    bound = 0.5 * ulp_f32(np.abs(theta) + S) + 0.5 * ulp_f32(theta)
    assert np.all(np.abs(t[0].astype(np.float64) - theta) <= bound)


def test_update_sequential_vs_fused():
    """K separate passes each round once; the fused update rounds once. The two
    differ by at most K half-ulps of the running value (fp32)."""
    seed, lr, K = 0x15E5A0006, 1e-3, 12
    c = np.random.default_rng(6).normal(0, 10, K)
    theta = W.tiny_theta(4096)
    t1, t2 = [theta.copy()], [theta.copy()]
    oracle.update(t1, [W.DT_F32], seed, c, lr)
    oracle.update_sequential(t2, [W.DT_F32], seed, c, lr)
    a = update_coeffs(c, lr).astype(np.float64)
    bound = (K + 1) * 0.5 * ulp_f32(np.abs(theta) + np.abs(a).sum())
    assert np.all(np.abs(t1[0].astype(np.float64) - t2[0]) <= bound)
    # sequential == K perturb passes exactly
    t3 = [theta.copy()]
    for k in range(K):
        oracle.perturb(t3, [W.DT_F32], seed, k, float(update_coeffs(c, lr)[k]))
    np.testing.assert_array_equal(t2[0], t3[0])


def test_update_descends_quadratic():
    """On the quadratic with many probes and alpha = 0, one 1.5-SPSA step at a
    small lr lowers the loss (SPSA's expected direction is -grad f)."""
    theta, a = quad_setup(d=2048, seed=3)
    eps, K, seed, lr = 2.0 ** -10, 64, 0x15E5A00AA, 2.0 ** -10
    t = [theta.copy()]
    L0 = oracle.quadratic_loss(t[0], a)
    rows = []
    for k in range(K):
        oracle.perturb(t, [W.DT_F32], seed, k, eps)
        lp = oracle.quadratic_loss(t[0], a)
        oracle.perturb(t, [W.DT_F32], seed, k, -2 * eps)
        lm = oracle.quadratic_loss(t[0], a)
        oracle.perturb(t, [W.DT_F32], seed, k, eps)
        rows.append([lp, lm, L0])
    rc, c, w, cv = oracle.precondition(rows, eps)
    oracle.update(t, [W.DT_F32], seed, c, lr * 0.05)
    assert oracle.quadratic_loss(t[0], a) < L0


def test_update_bad_args():
    with pytest.raises(RuntimeError):
        oracle.update([np.zeros(4, np.float32)], [W.DT_F32], 1, np.zeros(0), 1e-3)
    with pytest.raises(RuntimeError):
        oracle.update([np.zeros(4, np.float32)], [7], 1, np.ones(2), 1e-3)


# ------------------------------------------------------------------- loss
def test_quadratic_loss():
    n = 1000
    assert oracle.quadratic_loss(np.ones(n, np.float32), np.ones(n, np.float32)) == n / 2
    th = W.tiny_theta(10000)
    a = W.tiny_curvatures(10000)
    want = 0.5 * math.fsum(a.astype(np.float64) * th.astype(np.float64) ** 2)
    assert oracle.quadratic_loss(th, a) == pytest.approx(want, rel=1e-13)


@pytest.mark.parametrize("dtype", [W.DT_F32, W.DT_BF16, W.DT_F16])
def test_element_routines_match_list_routines(dtype):
    """The element-list routines (sampled full-size parity, the CPU baseline)
    compute what the tensor-list routines compute at the same virtual indices."""
    rng = np.random.default_rng(21)
    n = 3000
    bits = W.random_storage(rng, n, dtype)
    g = np.arange(n, dtype=np.uint64)
    seed, eps = 0x15E5A0004, 1e-3
    c = rng.standard_normal(12) * 3

    def widen(b):
        if dtype == W.DT_F32:
            return b
        if dtype == W.DT_F16:
            return b.view(np.float16).astype(np.float32)
        return (b.astype(np.uint32) << 16).view(np.float32)

    def narrow(out):
        return out.view(np.float32) if dtype == W.DT_F32 else out.astype(np.uint16)

    t = [bits.copy()]
    e = bits.copy()
    for k, s in ((0, eps), (5, -2 * eps), (9, 0.25)):
        oracle.perturb(t, [dtype], seed, k, s)
        e = narrow(oracle.perturb_elements(dtype, g, widen(e), seed, k, s))
        np.testing.assert_array_equal(e.view(np.uint8), t[0].view(np.uint8))
    oracle.update(t, [dtype], seed, c, 1e-2)
    e = narrow(oracle.update_elements(dtype, g, widen(e), seed, c, 1e-2))
    np.testing.assert_array_equal(e.view(np.uint8), t[0].view(np.uint8))
