"""Pins for the oracle's probe generator.

* Philox4x32-10 against Triton's independent implementation (CPU interpreter).
* The probe definition (block / group / byte / bit mapping and the unpack rule
  of Appendix F) against an independent route: Triton's Philox words viewed as
  little-endian bytes and unpacked with numpy.unpackbits(bitorder="little"),
  which is exactly "bit i%8 of byte i//8".
* Rademacher statistics: balance, probe/seed independence.
"""
import numpy as np
import pytest

import oracle

U32 = 0xFFFFFFFF


def test_philox_matches_triton(triton_philox):
    rng = np.random.default_rng(7)
    seeds = np.array([0, 1, 0x123456789ABCDEF, 0xFFFFFFFFFFFFFFFF, 0x15E5A0000, int(rng.integers(0, 2**63))],
                     dtype=np.uint64)
    N = 64
    ctr = rng.integers(0, 2**32, size=(len(seeds), N, 4), dtype=np.uint64).astype(np.uint32)
    ctr[:, 0, :] = 0
    ctr[:, 1, :] = U32
    ctr[:, 2, :] = [1, 0, 0, 0]
    ctr[:, 3, :] = [0, 0, 0, 1]
    ref = triton_philox(seeds, ctr)
    for s, seed in enumerate(seeds):
        key = [int(seed) & U32, int(seed) >> 32]
        for i in range(N):
            got = oracle.philox4x32_10(ctr[s, i], key)
            np.testing.assert_array_equal(got, ref[s, i], err_msg=f"seed={seed:#x} ctr={ctr[s, i]}")


def independent_signs(triton_philox, seed, k, g):
    """z_k[g] through Triton's Philox + numpy's little-endian bit unpacking."""
    g = np.asarray(g, dtype=np.uint64)
    blocks = g // np.uint64(16)
    N = 1
    while N < len(blocks):
        N *= 2
    ctr = np.zeros((1, N, 4), dtype=np.uint32)
    ctr[0, : len(blocks), 0] = (blocks & np.uint64(U32)).astype(np.uint32)
    ctr[0, : len(blocks), 1] = (blocks >> np.uint64(32)).astype(np.uint32)
    ctr[0, :, 2] = k // 8
    words = triton_philox([seed], ctr)[0, : len(blocks)]          # (n, 4) uint32
    by = np.ascontiguousarray(words.astype("<u4")).view(np.uint8).reshape(-1, 16)
    bits = np.unpackbits(by[:, :, None], axis=2, bitorder="little")  # (n, 16, 8)
    b = bits[np.arange(len(g)), (g % np.uint64(16)).astype(np.int64), k % 8]
    return b.astype(np.int8) * 2 - 1


@pytest.mark.parametrize("seed", [0x15E5A0003, 0xFFFFFFFFFFFFFFFF])
@pytest.mark.parametrize("k", [0, 5, 7, 8, 13, 255, 1023])
def test_probe_signs_independent_route(triton_philox, seed, k):
    rng = np.random.default_rng(k)
    g = np.concatenate([np.arange(0, 64), np.arange(2**32 * 16 - 8, 2**32 * 16 + 8),
                        rng.integers(0, 2**40, 200)]).astype(np.uint64)
    want = independent_signs(triton_philox, seed, k, g)
    got = np.array([oracle.probe_sign(seed, k, int(x)) for x in g], dtype=np.int8)
    np.testing.assert_array_equal(got, want)


def test_probe_bytes_unpack_rule():
    """Appendix F unpack: element i is bit i%8 of byte i//8, bit 1 -> +1."""
    seed, k = 0x15E5A0001, 11
    for first in (0, 3, 1000001):
        n = 300
        packed = oracle.probe_bytes(seed, k, first, n)
        signs = oracle.probe_signs(seed, k, 8 * first, 8 * n)
        unpacked = np.unpackbits(packed, bitorder="little").astype(np.int8) * 2 - 1
        np.testing.assert_array_equal(unpacked, signs)


def test_probe_balance_and_independence():
    n = 1 << 20
    seed = 0x15E5A0000
    z0 = oracle.probe_signs(seed, 0, 0, n).astype(np.float64)
    z1 = oracle.probe_signs(seed, 1, 0, n).astype(np.float64)
    z8 = oracle.probe_signs(seed, 8, 0, n).astype(np.float64)
    zs = oracle.probe_signs(seed + 1, 0, 0, n).astype(np.float64)
    sigma = 1.0 / np.sqrt(n)
    for z in (z0, z1, z8, zs):
        assert set(np.unique(z)) == {-1.0, 1.0}
        assert abs(z.mean()) < 5 * sigma
    for a, b in ((z0, z1), (z0, z8), (z0, zs), (z1, z8)):
        assert abs(np.mean(a * b)) < 5 * sigma
    # neighbouring elements (same byte, same word, next block) are uncorrelated
    for lag in (1, 8, 16, 128):
        assert abs(np.mean(z0[:-lag] * z0[lag:])) < 5 * sigma


def test_probe_bit_positions_balanced():
    """Each of the 8 probes sharing a byte, and each of the 16 byte slots of a
    block, sees a balanced sign."""
    seed = 0x15E5A0009
    n = 1 << 16
    for k in range(8):
        z = oracle.probe_signs(seed, k, 0, n).reshape(-1, 16).astype(np.float64)
        m = z.mean(axis=0)
        assert np.all(np.abs(m) < 5 / np.sqrt(z.shape[0]))


def test_virtual_offsets():
    numel = [0, 1, 16, 17, 31, 32, 5]
    want = [0, 0, 16, 32, 64, 96, 128]
    np.testing.assert_array_equal(oracle.virtual_offsets(numel), want)


def independent_signs_p8(triton_philox, seed, k, g):
    """Packing 8: z_k[g] = bit 0 of byte g mod 16 of Philox(g/16, k, 0)."""
    g = np.asarray(g, dtype=np.uint64)
    blocks = g // np.uint64(16)
    N = 1
    while N < len(blocks):
        N *= 2
    ctr = np.zeros((1, N, 4), dtype=np.uint32)
    ctr[0, : len(blocks), 0] = (blocks & np.uint64(U32)).astype(np.uint32)
    ctr[0, : len(blocks), 1] = (blocks >> np.uint64(32)).astype(np.uint32)
    ctr[0, :, 2] = k
    words = triton_philox([seed], ctr)[0, : len(blocks)]
    by = np.ascontiguousarray(words.astype("<u4")).view(np.uint8).reshape(-1, 16)
    b = by[np.arange(len(g)), (g % np.uint64(16)).astype(np.int64)] & 1
    return b.astype(np.int8) * 2 - 1


@pytest.mark.parametrize("k", [0, 3, 8, 1023])
def test_probe_signs_packing8_independent_route(triton_philox, k):
    import oracle as O
    seed = 0x15E5A0003
    rng = np.random.default_rng(k + 50)
    g = np.concatenate([np.arange(0, 64), rng.integers(0, 2**40, 200)]).astype(np.uint64)
    want = independent_signs_p8(triton_philox, seed, k, g)
    with O.packing(8):
        got = np.array([O.probe_sign(seed, k, int(x)) for x in g], dtype=np.int8)
    np.testing.assert_array_equal(got, want)


def test_packing8_balance_and_independence():
    import oracle as O
    n = 1 << 18
    seed = 0x15E5A0000
    with O.packing(8):
        zs = [O.probe_signs(seed, k, 0, n).astype(np.float64) for k in (0, 1, 7, 8)]
        packed = O.probe_bytes(seed, 5, 0, 1000)
        signs = O.probe_signs(seed, 5, 0, 8000)
    np.testing.assert_array_equal(np.unpackbits(packed, bitorder="little").astype(np.int8) * 2 - 1, signs)
    sigma = 1.0 / np.sqrt(n)
    for z in zs:
        assert abs(z.mean()) < 5 * sigma
    for a in range(4):
        for b in range(a + 1, 4):
            assert abs(np.mean(zs[a] * zs[b])) < 5 * sigma
    # the two packings define different probes
    z1 = oracle.probe_signs(seed, 1, 0, n).astype(np.float64)
    assert abs(np.mean(z1 * zs[1])) < 5 * sigma
