"""Special values on the device, against the oracle.

Weights: every bf16 and every fp16 bit pattern (signed zeros, subnormals,
the largest finite values, infinities, every NaN), and for fp32 storage the
same classes (NaNs with payloads, quiet and signalling) plus seeded random
bit patterns. Each list holds the patterns three times: an aligned tensor
(the 256-bit block path), a view one element in (the aligned-chunk kernels)
and a short tail (the element-wise path).

Scales: small and large ones of both signs, one that lands every weight of
[1, 2) exactly halfway between two storage values (round-to-nearest-even
ties), and one that carries the largest finite value past the format's
range. Perturbation passes (single, two-op, pair, Algorithm 1's sequential
update) are compared bit for bit; the fused update within one storage ulp
(outside the cancellation band) with NaNs in the same encoding. NaN results
are stored as the all-ones positive quiet NaN of the storage format (a
reading: the paper says nothing about NaN weights, and IEEE 754 leaves a NaN
result's sign and payload to the implementation).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

from gpu_helpers import assert_update_close, storage_bits, storage_np, to_torch

pytestmark = pytest.mark.gpu

ALL16 = np.arange(65536, dtype=np.uint32).astype(np.uint16)
F32_SPECIAL_BITS = [0x00000000, 0x80000000, 0x7F800000, 0xFF800000, 0x7FC00000, 0xFFC00000, 0x7FC00001,
                    0x7F800001, 0xFFBFFFFF, 0x7FFFFFFF, 0xFFFFFFFF, 0x00000001, 0x80000001, 0x007FFFFF,
                    0x807FFFFF, 0x00800000, 0x80800000, 0x7F7FFFFF, 0xFF7FFFFF, 0x7F7FFFFE, 0x3F800000,
                    0xBF800000, 0x3F800001, 0x33800000, 0x34000000]


def f32_patterns():
    rng = np.random.default_rng(17)
    rand = rng.integers(0, 2 ** 32, 1 << 16, dtype=np.uint64).astype(np.uint32)
    # weights of [1, 2) and near fp32's largest value, where the tie and overflow scales act
    ones = (np.uint32(0x3F800000) + rng.integers(0, 1 << 23, 4096, dtype=np.uint64).astype(np.uint32))
    top = np.uint32(0x7F7FFFFF) - np.arange(64, dtype=np.uint32)
    bits = np.concatenate([np.array(F32_SPECIAL_BITS, dtype=np.uint32), rand, ones, top, top | np.uint32(0x80000000)])
    return bits.view(np.float32)


CASES = {
    # dtype: (patterns, scales); the fourth scale makes ties in [1, 2), the last overflows
    "bf16": (W.DT_BF16, torch.bfloat16, ALL16, [1e-3, -1e-3, -0.5, 2.0 ** -8, -(2.0 ** -8), 2.0 ** 121]),
    "f16": (W.DT_F16, torch.float16, ALL16, [1e-3, -1e-3, 0.5, 2.0 ** -11, -(2.0 ** -11), 32.0]),
    "f32": (W.DT_F32, torch.float32, None, [1e-3, -0.5, 2.0 ** -24, -(2.0 ** -24), 2.0 ** 103, 2.0 ** 104]),
}


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def make(name):
    """Host storage arrays and device tensors: aligned, a view one element in,
    and a 21-element tail."""
    dt, tdt, pat, _ = CASES[name]
    pat = f32_patterns() if pat is None else pat
    host = [pat.copy(), pat[::-1].copy(), pat[1000:1021].copy()]
    a = to_torch(host[0], tdt)
    base = torch.empty(pat.size + 1, dtype=tdt, device="cuda")
    view = base[1:]
    view.copy_(to_torch(host[1], tdt))
    tail = to_torch(host[2], tdt)
    return host, [a, view, tail], dt


def assert_bits_equal(dev, host, what):
    for i, (d, h) in enumerate(zip(dev, host)):
        got, want = storage_bits(d), storage_bits(h)
        bad = np.nonzero(got != want)[0]
        assert bad.size == 0, (what, i, [(int(j), hex(int(storage_bits(h)[j])), hex(int(got[j])), hex(int(want[j])))
                                         for j in bad[:5]])


@pytest.mark.parametrize("name", list(CASES))
def test_perturb_special_values(name, packing_mode):
    seed = W.step_seed(41)
    for s_i, scale in enumerate(CASES[name][3]):
        host, dev, dt = make(name)
        ref = [h.copy() for h in host]
        zo.perturb(dev, seed, 3 + s_i, scale)
        oracle.perturb(host, [dt] * 3, seed, 3 + s_i, scale)
        assert_bits_equal(dev, host, f"{name} perturb scale {scale}")
        # the pattern really exercised what it should: some results changed
        assert any(np.any(storage_bits(d) != storage_bits(r)) for d, r in zip(dev, ref))


@pytest.mark.parametrize("name", list(CASES))
def test_perturb2_special_values(name):
    seed = W.step_seed(42)
    scales = CASES[name][3]
    for (ka, sa, kb, sb) in ((5, scales[3], 6, scales[5]), (7, scales[0], 8, scales[2])):
        host, dev, dt = make(name)
        zo.perturb2(dev, seed, ka, sa, kb, sb)
        oracle.perturb(host, [dt] * 3, seed, ka, sa)
        oracle.perturb(host, [dt] * 3, seed, kb, sb)
        assert_bits_equal(dev, host, f"{name} perturb2 ({ka}, {sa}) ({kb}, {sb})")


@pytest.mark.parametrize("name", list(CASES))
def test_pair_special_values(name):
    seed = W.step_seed(43)
    for scale in (CASES[name][3][3], CASES[name][3][5], 0.25):
        host, dev, dt = make(name)
        plus = [torch.empty_like(d) for d in dev]
        minus = [torch.empty_like(d) for d in dev]
        zo.perturb_pair(dev, plus, minus, seed, 9, scale)
        hp, hm = [h.copy() for h in host], [h.copy() for h in host]
        oracle.perturb(hp, [dt] * 3, seed, 9, scale)
        oracle.perturb(hm, [dt] * 3, seed, 9, -scale)
        assert_bits_equal(plus, hp, f"{name} pair plus {scale}")
        assert_bits_equal(minus, hm, f"{name} pair minus {scale}")
        assert_bits_equal(dev, host, f"{name} pair theta untouched")


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("K,pre", [(8, False), (64, True), (256, True)])
def test_update_special_values(name, K, pre, packing_mode):
    seed = W.step_seed(44)
    lr = 1e-2
    c_np = np.random.default_rng(K).normal(0, 5, K)
    c = torch.tensor(c_np, dtype=torch.float64, device="cuda")
    host, dev, dt = make(name)
    zo.update(dev, seed, c, lr, pre=(K - 1, 1e-3) if pre else None)
    if pre:
        oracle.perturb(host, [dt] * 3, seed, K - 1, 1e-3)
    oracle.update(host, [dt] * 3, seed, c_np, lr)
    for i, (d, h) in enumerate(zip(dev, host)):
        st = assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, lr, context=f"{name} K={K} tensor {i}")
        print(f"specials update {name} K={K} pre={pre} tensor {i}: {st}")


@pytest.mark.parametrize("name", list(CASES))
def test_update_sequential_special_values(name):
    seed = W.step_seed(45)
    c_np = np.random.default_rng(5).normal(0, 5, 5)
    c = torch.tensor(c_np, dtype=torch.float64, device="cuda")
    host, dev, dt = make(name)
    zo.update_sequential(dev, seed, c, 1e-2)
    oracle.update_sequential(host, [dt] * 3, seed, c_np, 1e-2)
    assert_bits_equal(dev, host, f"{name} sequential update")


def test_nan_encoding_is_the_canonical_one():
    """Every NaN weight comes back as 0x7FFF (16-bit) / 0x7FFFFFFF (fp32)."""
    for name in CASES:
        host, dev, dt = make(name)
        zo.perturb(dev, W.step_seed(46), 1, 1e-3)
        for d in dev:
            v = storage_np(d)
            b = storage_bits(d)
            f = v if v.dtype == np.float32 else None
            if f is None:
                nan = (b & 0x7FFF) > (0x7F80 if dt == W.DT_BF16 else 0x7C00)
                assert np.all(b[nan] == 0x7FFF)
            else:
                assert np.all(b[np.isnan(f)] == 0x7FFFFFFF)
