"""Pins for the oracle's storage-format rounding: its IEEE-754 encoders must
agree bit for bit with numpy's float16 cast and torch's bfloat16 cast (both
round to nearest, ties to even) on random values and on every edge case."""
import numpy as np
import pytest
import torch

import oracle


def edge_values():
    v = [0.0, -0.0, 1.0, -1.0, 65504.0, 65519.99, 65520.0, 65536.0, 1e30, -1e30, 3.4e38,
         2.0 ** -14, 2.0 ** -24, 2.0 ** -25, 2.0 ** -25 * 1.5, 2.0 ** -26, 2.0 ** -15 * 1.0009765625,
         1.0 + 2.0 ** -11, 1.0 + 3 * 2.0 ** -11, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -8 + 2.0 ** -20,
         2.0 ** -126, 2.0 ** -133, 2.0 ** -134, 2.0 ** -149, 3.3895313892515355e38, 3.3961e38,
         float("inf"), float("-inf")]
    return np.array(v, dtype=np.float32)


def random_values(n=20000, seed=3):
    rng = np.random.default_rng(seed)
    bits = rng.integers(0, 2**32, n, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    y = (rng.standard_normal(n) * 0.02).astype(np.float32)
    return np.concatenate([x, y, edge_values()])


def test_f16_matches_numpy():
    x = random_values()
    with np.errstate(over="ignore"):          # overflow to inf is one of the cases checked
        want = x.astype(np.float16).view(np.uint16)
    got = oracle.f32_to_f16(x)
    bad = np.nonzero(got != want)[0]
    assert bad.size == 0, [(float(x[i]), hex(got[i]), hex(want[i])) for i in bad[:5]]


def test_f16_decode_matches_numpy():
    h = np.arange(0, 65536, dtype=np.uint32).astype(np.uint16)
    want = h.view(np.float16).astype(np.float32)
    got = oracle.f16_to_f32(h)
    fin = np.isfinite(want)
    np.testing.assert_array_equal(got[fin].view(np.uint32), want[fin].view(np.uint32))
    assert np.all(np.isnan(got[~fin]) == np.isnan(want[~fin]))


def test_bf16_matches_torch():
    x = random_values()
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.f32_to_bf16(x)
    bad = np.nonzero(got != want)[0]
    assert bad.size == 0, [(float(x[i]), hex(got[i]), hex(want[i])) for i in bad[:5]]


def test_bf16_decode_matches_torch():
    h = np.arange(0, 65536, dtype=np.uint32).astype(np.uint16)
    want = torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).float().numpy()
    got = oracle.bf16_to_f32(h)
    fin = np.isfinite(want)
    np.testing.assert_array_equal(got[fin].view(np.uint32), want[fin].view(np.uint32))


@pytest.mark.parametrize("enc", [oracle.f32_to_f16, oracle.f32_to_bf16])
def test_nan_stays_nan(enc):
    h = enc(np.array([np.nan], dtype=np.float32))[0]
    dec = oracle.f16_to_f32 if enc is oracle.f32_to_f16 else oracle.bf16_to_f32
    assert np.isnan(dec(np.array([h], dtype=np.uint16))[0])


# ------------------------------------------------------------ special values
# The oracle's perturbation and update of every 16-bit pattern (and of fp32
# specials) against numpy's own IEEE arithmetic and casts. NaN results: the
# oracle stores the all-ones positive quiet NaN (0x7FFF, 0x7FFFFFFF), a
# reading -- IEEE 754 leaves a NaN result's sign and payload open -- so numpy
# pins only that they are NaN.
ALL16 = np.arange(65536, dtype=np.uint32).astype(np.uint16)
F32_SPECIALS = np.array([0x00000000, 0x80000000, 0x7F800000, 0xFF800000, 0x7FC00000, 0xFFC00001, 0x7F800001,
                         0x00000001, 0x807FFFFF, 0x00800000, 0x7F7FFFFF, 0xFF7FFFFF, 0x3F800000, 0x3F800001],
                        dtype=np.uint32).view(np.float32)


def widen16(bits, dt):
    if dt == oracle.F16:
        return bits.view(np.float16).astype(np.float32)
    return (bits.astype(np.uint32) << 16).view(np.float32)


def narrow16(x, dt):
    if dt == oracle.F16:
        with np.errstate(over="ignore"):
            return x.astype(np.float16).view(np.uint16)
    return torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("dt", [oracle.BF16, oracle.F16])
@pytest.mark.parametrize("scale", [1e-3, -0.5, 2.0 ** -8, 2.0 ** -11, 32.0, 2.0 ** 121])
def test_perturb_every_16bit_pattern_against_numpy(dt, scale):
    seed, k = 0x15E5A0007, 11
    z = oracle.probe_signs(seed, k, 0, ALL16.size).astype(np.float32)
    host = [ALL16.copy()]
    oracle.perturb(host, [dt], seed, k, scale)
    with np.errstate(over="ignore", invalid="ignore"):
        r = widen16(ALL16, dt) + np.float32(scale) * z
    want = narrow16(r, dt)
    nan = np.isnan(r)
    np.testing.assert_array_equal(host[0][~nan], want[~nan])
    assert np.all(host[0][nan] == 0x7FFF)
    exp_mask = 0x7F80 if dt == oracle.BF16 else 0x7C00
    assert np.sum(nan) == np.sum(((ALL16 & exp_mask) == exp_mask) & ((ALL16 & ~np.uint16(exp_mask) & 0x7FFF) != 0))


@pytest.mark.parametrize("scale", [1e-3, -0.5, 2.0 ** -24, 2.0 ** 103, 2.0 ** 104])
def test_perturb_fp32_specials_against_numpy(scale):
    seed, k = 0x15E5A0007, 3
    rng = np.random.default_rng(5)
    x = np.concatenate([F32_SPECIALS, rng.integers(0, 2 ** 32, 4096, dtype=np.uint64).astype(np.uint32)
                        .view(np.float32)])
    z = oracle.probe_signs(seed, k, 0, x.size).astype(np.float32)
    host = [x.copy()]
    oracle.perturb(host, [oracle.F32], seed, k, scale)
    with np.errstate(over="ignore", invalid="ignore"):
        r = x + np.float32(scale) * z
    nan = np.isnan(r)
    np.testing.assert_array_equal(host[0].view(np.uint32)[~nan], r.view(np.uint32)[~nan])
    assert np.all(host[0].view(np.uint32)[nan] == 0x7FFFFFFF) and nan.any()


@pytest.mark.parametrize("dt", [oracle.F16, oracle.F32])
def test_update_specials_against_numpy_fp64(dt):
    """Fused update: theta + sum_k a_k z_k formed exactly in fp64 by numpy and
    rounded once by numpy's own cast (fp64 -> fp16 / fp32 in one rounding)."""
    seed, K, lr = 0x15E5A0008, 16, 1e-2
    c = np.random.default_rng(8).normal(0, 5, K)
    x = ALL16.copy() if dt == oracle.F16 else np.concatenate([F32_SPECIALS, (np.random.default_rng(6).standard_normal(
        4096) * 0.02).astype(np.float32)])
    n = x.size
    a = np.array([np.float32(-(lr / K) * ck) for ck in c], dtype=np.float64)
    A = np.zeros(n)
    for k in range(K):
        A += a[k] * oracle.probe_signs(seed, k, 0, n).astype(np.float64)
    host = [x.copy()]
    oracle.update(host, [dt], seed, c, lr)
    with np.errstate(over="ignore", invalid="ignore"):
        th = x.view(np.float16).astype(np.float64) if dt == oracle.F16 else x.astype(np.float64)
        v = th + A
        want = v.astype(np.float16).view(np.uint16) if dt == oracle.F16 else v.astype(np.float32).view(np.uint32)
    got = host[0] if dt == oracle.F16 else host[0].view(np.uint32)
    nan = np.isnan(v)
    np.testing.assert_array_equal(got[~nan], want[~nan])
    assert np.all(got[nan] == (0x7FFF if dt == oracle.F16 else 0x7FFFFFFF)) and nan.any()


def test_update_bf16_specials():
    """bf16: infinities stay infinite and every NaN comes back as 0x7FFF."""
    seed, K = 0x15E5A0009, 8
    host = [ALL16.copy()]
    oracle.update(host, [oracle.BF16], seed, np.ones(K), 1e-3)
    inf = (ALL16 & 0x7FFF) == 0x7F80
    nan = (ALL16 & 0x7FFF) > 0x7F80
    np.testing.assert_array_equal(host[0][inf], ALL16[inf])
    assert np.all(host[0][nan] == 0x7FFF)
