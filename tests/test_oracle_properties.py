"""Property-based pins of the oracle (hypothesis): the storage encoders over
arbitrary fp32 bit patterns against numpy / torch casts, the perturbation's
arithmetic against numpy's IEEE fp32 addition, and invariants of the
preconditioner and the fused update that hold for any input."""
import numpy as np
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import given, settings  # noqa: E402
from hypothesis import strategies as st  # noqa: E402

import oracle  # noqa: E402
from paper_2609_38095_gb300 import workloads as W  # noqa: E402

SETTINGS = settings(max_examples=300, deadline=None)
u32 = st.integers(min_value=0, max_value=2**32 - 1)


def as_f32(bits):
    return np.array([bits], dtype=np.uint32).view(np.float32)[0]


@SETTINGS
@given(bits=u32)
def test_f32_to_f16_any_pattern(bits):
    x = as_f32(bits)
    got = int(oracle.f32_to_f16(np.array([x]))[0])
    with np.errstate(over="ignore"):
        want = int(np.array([x], dtype=np.float32).astype(np.float16).view(np.uint16)[0])
    if np.isnan(x):
        assert (got & 0x7C00) == 0x7C00 and (got & 0x3FF) != 0
    else:
        assert got == want


@SETTINGS
@given(bits=u32)
def test_f32_to_bf16_any_pattern(bits):
    torch = pytest.importorskip("torch")
    x = as_f32(bits)
    got = int(oracle.f32_to_bf16(np.array([x]))[0])
    want = int(torch.tensor([x], dtype=torch.float32).to(torch.bfloat16).view(torch.int16).item()) & 0xFFFF
    if np.isnan(x):
        assert (got & 0x7F80) == 0x7F80 and (got & 0x7F) != 0
    else:
        assert got == want


def finite_f32(min_abs=0.0, max_abs=1e30):
    return st.floats(min_value=-max_abs, max_value=max_abs, allow_nan=False, allow_infinity=False,
                     width=32).filter(lambda v: abs(v) >= min_abs)


@SETTINGS
@given(theta=finite_f32(max_abs=1e6), scale=finite_f32(max_abs=10.0), k=st.integers(0, 1023),
       g=st.integers(0, 2**40), dt=st.sampled_from([W.DT_F32, W.DT_BF16, W.DT_F16]))
def test_perturb_element_is_one_fp32_add_and_one_rounding(theta, scale, k, g, dt):
    """theta' = rn_storage(fl32(theta + scale * z)), with fl32 numpy's IEEE
    addition and rn_storage numpy's / torch's cast."""
    th = np.float32(theta)
    if dt == W.DT_BF16:
        th = (np.array([th]).view(np.uint32) & 0xFFFF0000).view(np.float32)[0]   # a bf16 value
    elif dt == W.DT_F16:
        with np.errstate(over="ignore"):
            th = np.float32(np.float16(th)) if np.isfinite(np.float16(th)) else np.float32(0.0)
    seed = 0x15E5A0000 + k
    z = oracle.probe_sign(seed, k, g)
    out = int(oracle.perturb_elements(dt, [g], [th], seed, k, scale)[0])
    s = np.float32(np.float32(scale) * np.float32(z))
    r = np.float32(th + s)
    if dt == W.DT_F32:
        assert out == int(np.array([r]).view(np.uint32)[0])
    elif dt == W.DT_F16:
        with np.errstate(over="ignore"):
            assert out == int(np.array([r]).astype(np.float16).view(np.uint16)[0])
    else:
        torch = pytest.importorskip("torch")
        want = int(torch.tensor([r], dtype=torch.float32).to(torch.bfloat16).view(torch.int16).item()) & 0xFFFF
        assert out == want


triples = st.lists(st.tuples(st.floats(-50, 50), st.floats(-50, 50), st.floats(-50, 50)), min_size=1, max_size=40)


@SETTINGS
@given(L=triples, eps=st.floats(1e-4, 1e-1), alpha=st.floats(0.0, 1.0), lam=st.floats(1e-3, 10.0),
       one_sided=st.booleans(), relative=st.booleans())
def test_precondition_invariants(L, eps, alpha, lam, one_sided, relative):
    """Any finite triples: 0 < w <= 1/lambda_reg; c carries the sign of the
    difference it scales and is at most |difference| / lambda_reg; without
    the relative flag a larger |curvature| never gives a larger weight."""
    L = np.array(L, dtype=np.float64)
    rc, c, w, cv = oracle.precondition(L, eps, alpha=alpha, lambda_reg=lam, one_sided=one_sided, relative=relative)
    assert rc == oracle.OK
    assert np.all(w > 0) and np.all(w <= 1.0 / lam * (1 + 1e-15))
    d = (L[:, 0] - L[:, 2]) / eps if one_sided else (L[:, 0] - L[:, 1]) / (2 * eps)
    assert np.all(np.sign(c) == np.sign(d) * (w > 0))
    assert np.all(np.abs(c) <= np.abs(d) / lam * (1 + 1e-12))
    if not relative:
        order = np.argsort(np.abs(cv), kind="stable")
        assert np.all(np.diff(w[order]) <= 1e-15 * w[order][1:])


@SETTINGS
@given(K=st.integers(1, 40), seed=st.integers(0, 2**64 - 1), cscale=st.floats(1e-3, 1e3),
       dt=st.sampled_from([W.DT_F32, W.DT_BF16, W.DT_F16]))
def test_update_from_zero_is_odd_in_the_coefficients(K, seed, cscale, dt):
    """From theta = 0 the update is one rounding of sum_k a_k z_k, so c and -c
    give results of equal magnitude and opposite sign (round to nearest even
    is symmetric)."""
    rng = np.random.default_rng(seed % 2**32)
    c = rng.standard_normal(K) * cscale
    n = 64
    zero = np.zeros(n, dtype=np.float32) if dt == W.DT_F32 else np.zeros(n, dtype=np.uint16)
    a, b = [zero.copy()], [zero.copy()]
    oracle.update(a, [dt], seed, c, 1e-3)
    oracle.update(b, [dt], seed, -c, 1e-3)
    if dt == W.DT_F32:
        np.testing.assert_array_equal(a[0], -b[0])
    else:
        sign = np.uint16(0x8000)
        nz = (a[0] & np.uint16(0x7FFF)) != 0
        np.testing.assert_array_equal(a[0][nz] ^ sign, b[0][nz])
        np.testing.assert_array_equal(a[0] & np.uint16(0x7FFF), b[0] & np.uint16(0x7FFF))
