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
