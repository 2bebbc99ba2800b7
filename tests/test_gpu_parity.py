"""GPU parity: every entry point of libzo.so, called through the C ABI, against
the CPU oracle on the same seeded inputs, element by element.

Bars: probe bytes / signs and perturb bit-exact; the fused update within one
ulp of the storage dtype for bf16/fp16 and within the derived fp32 bound for
fp32 storage; the preconditioner within 1e-6 relative; the quadratic loss
within 1e-12 relative.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

from gpu_helpers import (TORCH_TO_DT, assert_update_close, bits_to_f64, storage_bits, storage_np, to_torch,
                         ulp_distance16)

pytestmark = pytest.mark.gpu

DTS = [torch.float32, torch.bfloat16, torch.float16]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def make_list(numels, dtypes, seed=0):
    rng = np.random.default_rng(seed)
    host = [W.random_storage(rng, n, TORCH_TO_DT[dt]) for n, dt in zip(numels, dtypes)]
    dev = [to_torch(h, dt) for h, dt in zip(host, dtypes)]
    return host, dev


MIXED_NUMELS = [1, 15, 16, 17, 31, 33, 0, 255, 4096, 4099, 100003, 7, 65536 + 5]
MIXED_DTYPES = [DTS[i % 3] for i in range(len(MIXED_NUMELS))]


def assert_storage_equal(dev, host, what=""):
    for i, (d, h) in enumerate(zip(dev, host)):
        got = storage_np(d)
        assert got.dtype == h.dtype
        np.testing.assert_array_equal(got.view(np.uint32 if h.dtype == np.float32 else np.uint16),
                                      h.view(np.uint32 if h.dtype == np.float32 else np.uint16),
                                      err_msg=f"{what} tensor {i} numel {h.size}")


# -------------------------------------------------------------- probe views
@pytest.mark.parametrize("seed", [W.step_seed(0), 0xFFFFFFFFFFFFFFFF, 0])
@pytest.mark.parametrize("probe", [0, 7, 8, 255, 1023, 5000])
@pytest.mark.parametrize("first,n", [(0, 4096), (3, 1001), (2**33 + 5, 777)])
def test_probe_bytes_bit_exact(seed, probe, first, n, packing_mode):
    got = zo.probe_bytes(seed, probe, first, n).cpu().numpy()
    want = oracle.probe_bytes(seed, probe, first, n)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("seed", [W.step_seed(3), 0xFFFFFFFFFFFFFFFF])
@pytest.mark.parametrize("probe", [0, 5, 9, 1023])
@pytest.mark.parametrize("first,n", [(0, 5000), (13, 333), (2**36 + 1, 1000)])
def test_probe_signs_bit_exact(seed, probe, first, n, packing_mode):
    got = zo.probe_signs(seed, probe, first, n).cpu().numpy()
    want = oracle.probe_signs(seed, probe, first, n)
    np.testing.assert_array_equal(got, want)


# ------------------------------------------------------------------ perturb
def test_perturb_bit_exact_mixed_sequence(packing_mode):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES)
    plist = zo.ParamList(dev)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    seed, eps = W.step_seed(1), 1e-3
    for k in (0, 5, 8, 13):
        for s in (eps, -2 * eps, eps):
            zo.perturb(plist, seed, k, s)
            oracle.perturb(host, dts, seed, k, s)
            assert_storage_equal(dev, host, f"probe {k} scale {s}")


@pytest.mark.parametrize("scale", [0.5, -3e-8, 0.0, 1e4])
def test_perturb_bit_exact_scales(scale):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=4)
    zo.perturb(dev, W.step_seed(9), 3, scale)
    oracle.perturb(host, [TORCH_TO_DT[d] for d in MIXED_DTYPES], W.step_seed(9), 3, scale)
    assert_storage_equal(dev, host, f"scale {scale}")


@pytest.mark.parametrize("dtype", DTS)
@pytest.mark.parametrize("offset", [1, 2, 4, 8, 16])
def test_perturb_unaligned_views(dtype, offset):
    """Views at element offsets that break 32-byte alignment take the
    aligned-chunk path; results are identical."""
    rng = np.random.default_rng(offset)
    n = 4096 + 37
    base_host = W.random_storage(rng, n + offset + 64, TORCH_TO_DT[dtype])
    base = to_torch(base_host, dtype)
    view = base[offset:offset + n]
    host = [base_host[offset:offset + n].copy()]
    zo.perturb([view], W.step_seed(2), 11, 1e-3)
    oracle.perturb(host, [TORCH_TO_DT[dtype]], W.step_seed(2), 11, 1e-3)
    assert_storage_equal([view], host, f"offset {offset}")
    # everything outside the view is untouched
    after = storage_np(base)
    np.testing.assert_array_equal(after[:offset], base_host[:offset])
    np.testing.assert_array_equal(after[offset + n:], base_host[offset + n:])


SHIFT_SIZES = [1, 3, 14, 15, 16, 17, 31, 100, 4096 + 37, 20011]


def unaligned_list(dtype, seed, prefix=0):
    """A view at every element offset that breaks 32-byte alignment (sizes
    from under one 16-element chunk to several chunk groups), each in its own
    allocation with guard elements around it, an aligned tensor after each,
    optionally after `prefix` small aligned tensors (pushing the views into a
    later launch)."""
    per = 32 // torch.tensor([], dtype=dtype).element_size()
    rng = np.random.default_rng(seed)
    dt = TORCH_TO_DT[dtype]
    bases, views, host = [], [], []
    for _ in range(prefix):
        h = W.random_storage(rng, int(rng.integers(0, 40)), dt)
        views.append(to_torch(h, dtype))
        host.append(h.copy())
    for off in range(1, per):
        n = SHIFT_SIZES[off % len(SHIFT_SIZES)]
        bh = W.random_storage(rng, off + n + 40, dt)
        b = to_torch(bh, dtype)
        bases.append((bh, b, off, n))
        views.append(b[off:off + n])
        host.append(bh[off:off + n].copy())
        ah = W.random_storage(rng, 16 * off + 5, dt)
        views.append(to_torch(ah, dtype))
        host.append(ah.copy())
    return bases, views, host


def assert_guards(bases):
    for bh, b, off, n in bases:
        after = storage_np(b)
        np.testing.assert_array_equal(after[:off], bh[:off], err_msg=f"before the view at offset {off}")
        np.testing.assert_array_equal(after[off + n:], bh[off + n:], err_msg=f"after the view at offset {off}")


@pytest.mark.parametrize("dtype", DTS)
@pytest.mark.parametrize("ops", ["one", "two_same_group", "two_groups"])
@pytest.mark.parametrize("prefix", [0, 1030])
def test_perturb_every_unaligned_offset(dtype, ops, prefix, packing_mode):
    """Unaligned views are perturbed in 32-byte aligned chunks that straddle
    two Philox blocks: every offset, every size class, one and two
    operations (probes in one sign group and in two), in the first and in a
    later launch: bit for bit the oracle, nothing outside the views written."""
    bases, views, host = unaligned_list(dtype, seed=60 + prefix, prefix=prefix)
    dts = [TORCH_TO_DT[dtype]] * len(views)
    seed = W.step_seed(21)
    if ops == "one":
        zo.perturb(views, seed, 13, 1e-3)
        oracle.perturb(host, dts, seed, 13, 1e-3)
    else:
        k2 = 14 if ops == "two_same_group" else 22
        zo.perturb2(views, seed, 13, 1e-3, k2, -2e-3)
        oracle.perturb(host, dts, seed, 13, 1e-3)
        oracle.perturb(host, dts, seed, k2, -2e-3)
    assert_storage_equal(views, host, ops)
    assert_guards(bases)


@pytest.mark.parametrize("dtype", DTS)
@pytest.mark.parametrize("K", [5, 16, 64])
@pytest.mark.parametrize("pre", [False, True])
def test_update_every_unaligned_offset(dtype, K, pre, packing_mode):
    """The fused update of unaligned views (aligned chunks, probe sums taken
    from the neighbouring lane) gives bit for bit what update_kernel gives
    for the same values in aligned tensors, is within the derived bound of
    the oracle, and writes nothing outside the views."""
    bases, views, host = unaligned_list(dtype, seed=80 + K)
    dts = [TORCH_TO_DT[dtype]] * len(views)
    aligned = [to_torch(h.copy(), dtype) for h in host]
    c_np = np.random.default_rng(81 + K).normal(0, 25, K)
    c = torch.tensor(c_np, device="cuda")
    seed, lr = W.step_seed(6), 1e-3
    p = (K - 1, 1e-3) if pre else None
    zo.update(views, seed, c, lr, pre=p)
    zo.update(aligned, seed, c, lr, pre=p)
    for i, (x, y) in enumerate(zip(views, aligned)):
        assert torch.equal(x.contiguous().view(torch.uint8), y.view(torch.uint8)), f"tensor {i}"
    if pre:
        oracle.perturb(host, dts, seed, K - 1, 1e-3)
    oracle.update(host, dts, seed, c_np, lr)
    for i, (d, h) in enumerate(zip(views, host)):
        assert_update_close(storage_bits(d), storage_bits(h), TORCH_TO_DT[dtype], c_np, lr, context=f"tensor {i}")
    assert_guards(bases)


def test_update_unaligned_failed_preconditioner():
    """status != 0: the update kernels of unaligned views apply only the
    leading perturbation (or nothing without one)."""
    bases, views, host = unaligned_list(torch.bfloat16, seed=90)
    dts = [W.DT_BF16] * len(views)
    st = torch.tensor([zo.ZO_ERR_NONFINITE], dtype=torch.int32, device="cuda")
    c = torch.ones(8, dtype=torch.float64, device="cuda")
    seed = W.step_seed(8)
    zo.update(views, seed, c, 1e-3, status=st)
    assert_storage_equal(views, host, "no pre, failed status: untouched")
    zo.update(views, seed, c, 1e-3, status=st, pre=(3, 2e-3))
    oracle.perturb(host, dts, seed, 3, 2e-3)
    assert_storage_equal(views, host, "failed status: only the leading perturbation")
    assert_guards(bases)


@pytest.mark.parametrize("dtype", DTS)
def test_update_sequential_unaligned_views(dtype, packing_mode):
    """The comparator's per-probe passes read their scale from the device
    coefficients in the unaligned-chunk kernel too."""
    bases, views, host = unaligned_list(dtype, seed=70)
    dts = [TORCH_TO_DT[dtype]] * len(views)
    c_np = np.random.default_rng(71).normal(0, 25, 9)
    zo.update_sequential(views, W.step_seed(5), torch.tensor(c_np, device="cuda"), 2e-3)
    oracle.update_sequential(host, dts, W.step_seed(5), c_np, 2e-3)
    assert_storage_equal(views, host)
    assert_guards(bases)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float16])
@pytest.mark.parametrize("offset", [1, 2, 8])
def test_update_unaligned_views(dtype, offset):
    """Fused update (with a leading perturbation) on views 2-, 4- and
    16-byte aligned: within the update tolerance of the oracle, nothing
    outside the view written."""
    rng = np.random.default_rng(40 + offset)
    n = 4096 * 3 + 21
    dt = TORCH_TO_DT[dtype]
    base_host = W.random_storage(rng, n + offset + 40, dt)
    base = to_torch(base_host, dtype)
    view = base[offset:offset + n]
    host = [base_host[offset:offset + n].copy()]
    K, seed, lr = 24, W.step_seed(41), 1e-3
    c_np = rng.normal(0, 20, K)
    zo.update([view], seed, torch.tensor(c_np, device="cuda"), lr, pre=(K - 1, 1e-3))
    oracle.perturb(host, [dt], seed, K - 1, 1e-3)
    oracle.update(host, [dt], seed, c_np, lr)
    assert_update_close(storage_bits(view), storage_bits(host[0]), dt, c_np, lr, context=f"offset {offset}")
    after = storage_np(base)
    np.testing.assert_array_equal(after[:offset], base_host[:offset])
    np.testing.assert_array_equal(after[offset + n:], base_host[offset + n:])


def test_perturb_many_tensors_split_launches(packing_mode):
    """More tensors than one launch's table holds (1024)."""
    rng = np.random.default_rng(12)
    numels = [int(x) for x in rng.integers(0, 300, 2500)]
    dtypes = [DTS[int(x)] for x in rng.integers(0, 3, 2500)]
    host, dev = make_list(numels, dtypes, seed=12)
    dts = [TORCH_TO_DT[d] for d in dtypes]
    zo.perturb(dev, W.step_seed(5), 17, -2e-3)
    oracle.perturb(host, dts, W.step_seed(5), 17, -2e-3)
    assert_storage_equal(dev, host)
    c = torch.tensor(rng.normal(0, 20, 9), dtype=torch.float64, device="cuda")
    zo.update(dev, W.step_seed(5), c, 1e-3)
    oracle.update(host, dts, W.step_seed(5), c.cpu().numpy(), 1e-3)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c.cpu().numpy(), 1e-3)


def test_guard_bands_untouched():
    """Tensors carved out of one buffer with canaries between them."""
    numels = [17, 4096, 33, 1000]
    gap = 64
    total = sum(numels) + gap * (len(numels) + 1)
    buf = torch.full((total,), 7.0, dtype=torch.bfloat16, device="cuda")
    views, pos = [], gap
    for n in numels:
        views.append(buf[pos:pos + n])
        pos += n + gap
    for v in views:
        v.normal_(0, 0.02)
    canary_mask = torch.ones(total, dtype=torch.bool)
    pos = gap
    for n in numels:
        canary_mask[pos:pos + n] = False
        pos += n + gap
    zo.perturb(views, W.step_seed(0), 1, 1e-3)
    c = torch.linspace(-30, 30, 37, dtype=torch.float64, device="cuda")
    zo.update(views, W.step_seed(0), c, 1e-3)
    zo.update_sequential(views, W.step_seed(0), c[:5].contiguous(), 1e-3)
    assert torch.all(buf.cpu()[canary_mask] == 7.0)


def test_empty_and_zero_length():
    zo.perturb([], 1, 0, 1e-3)
    zo.update([], 1, torch.ones(3, dtype=torch.float64, device="cuda"), 1e-3)
    z = torch.empty(0, dtype=torch.bfloat16, device="cuda")
    host, dev = make_list([0, 5, 0], [torch.bfloat16] * 3)
    zo.perturb([z] + dev, 1, 0, 1e-3)
    oracle.perturb([np.zeros(0, np.uint16)] + host, [W.DT_BF16] * 4, 1, 0, 1e-3)
    assert_storage_equal(dev, host)


def test_lists_with_their_own_packing_in_one_process():
    """Two parameter lists naming different probe packings, used in turn in
    one process: each follows its own packing whatever the process default."""
    dts_t = [torch.bfloat16, torch.float32, torch.float16]
    host8, dev8 = make_list([4099, 333, 16], dts_t, seed=808)
    host1, dev1 = make_list([4099, 333, 16], dts_t, seed=808)
    dts = [TORCH_TO_DT[d] for d in dts_t]
    l8, l1 = zo.ParamList(dev8, packing=8), zo.ParamList(dev1, packing=1)
    seed, K = W.step_seed(808), 12
    c_np = np.random.default_rng(808).normal(0, 5, K)
    c = torch.tensor(c_np, device="cuda")
    with zo.packing(8):                       # the default names neither list's packing
        zo.perturb(l1, seed, 9, 1e-3)
        zo.perturb2(l1, seed, 3, 1e-3, 11, -1e-3)
        zo.update(l1, seed, c, 1e-2, pre=(K - 1, 1e-3))
    with zo.packing(1):
        zo.perturb(l8, seed, 9, 1e-3)
        zo.perturb2(l8, seed, 3, 1e-3, 11, -1e-3)
        zo.update(l8, seed, c, 1e-2, pre=(K - 1, 1e-3))
    for host, bits in ((host8, 8), (host1, 1)):
        with oracle.packing(bits):
            oracle.perturb(host, dts, seed, 9, 1e-3)
            oracle.perturb(host, dts, seed, 3, 1e-3)
            oracle.perturb(host, dts, seed, 11, -1e-3)
            oracle.perturb(host, dts, seed, K - 1, 1e-3)
            oracle.update(host, dts, seed, c_np, 1e-2)
    for dev, host in ((dev8, host8), (dev1, host1)):
        for i, (d, h, dt) in enumerate(zip(dev, host, dts)):
            assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, 1e-2, context=f"tensor {i}")
    # the two packings give different probes: the lists really differ
    assert not np.array_equal(storage_bits(dev8[0]), storage_bits(dev1[0]))


# ------------------------------------------------------------------- update
@pytest.mark.parametrize("K", [1, 3, 8, 13, 64, 256])
def test_update_within_tolerance(K, packing_mode):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=K)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    rng = np.random.default_rng(100 + K)
    c_np = rng.normal(0, 25, K)
    c = torch.tensor(c_np, dtype=torch.float64, device="cuda")
    lr, seed = 1e-3, W.step_seed(K)
    zo.update(dev, seed, c, lr)
    oracle.update(host, dts, seed, c_np, lr)
    for i, (d, h, dt) in enumerate(zip(dev, host, dts)):
        st = assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, lr, context=f"K={K} tensor {i}")
        if dt != W.DT_F32:
            print(f"K={K} tensor {i}: {st}")


@pytest.mark.parametrize("bpt,K,pre", [(8, 24, True), (8, 40, False), (4, 24, False), (4, 40, True),
                                       (2, 64, True), (2, 200, False)])
def test_update_every_chunk_size(bpt, K, pre):
    """The 8-probe-table update (packing 1, 16 < K <= 384) gives each CTA a
    chunk of 512 x BPT blocks, BPT = 8, 4 or 2 by launch size (every SM gets
    a chunk). Lists sized for each BPT on this device, with bf16, fp16 and
    fp32 tensors, partial last blocks, a zero-length tensor and a view off the
    32-byte grid (its blocks skipped by the kernel and done by
    update_shift_kernel), against the oracle element by element."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    blocks = sms * 512 * bpt + 3 * 512 + 7            # just above this BPT's threshold
    numels = [blocks * 16 - 9 * 4096 - 3001 - 17, 4096 * 9 + 5, 0, 3001, 17]
    dtypes = [torch.bfloat16, torch.float16, torch.bfloat16, torch.float32, torch.float16]
    host, dev = make_list(numels, dtypes, seed=bpt * 1000 + K)
    # the fp16 tensor as a view one element into its own allocation
    base = torch.empty(numels[1] + 1, dtype=torch.float16, device="cuda")
    dev[1] = base[1:]
    dev[1].copy_(to_torch(host[1], torch.float16))
    dts = [TORCH_TO_DT[d] for d in dtypes]
    c_np = np.random.default_rng(K + bpt).normal(0, 25, K)
    c = torch.tensor(c_np, dtype=torch.float64, device="cuda")
    seed, lr, eps = W.step_seed(K + bpt), 1e-3, 1e-3
    zo.update(dev, seed, c, lr, pre=(K - 1, eps) if pre else None)
    if pre:
        oracle.perturb(host, dts, seed, K - 1, eps)
    oracle.update(host, dts, seed, c_np, lr)
    for i, (d, h, dt) in enumerate(zip(dev, host, dts)):
        if h.size:
            st = assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, lr,
                                     context=f"BPT={bpt} K={K} tensor {i}")
            print(f"BPT={bpt} K={K} tensor {i}: {st}")


@pytest.mark.parametrize("n_alias", [32, 45])
def test_perturb_beyond_2_32_blocks(n_alias):
    """The perturbation passes on tensors whose Philox block counter has a
    non-zero high word (virtual index >= 2^36), laid out as in
    test_update_beyond_2_32_blocks: with 32 aliased 2^31-element entries in
    front, the checked tensors' launch straddles block 2^32; with 45 it
    starts above it. A single pass, a two-op pass in one group of 8 and one
    across two groups (the two-group kernel), each bit-exact with the oracle
    at the checked tensors' virtual indices."""
    free, _ = torch.cuda.mem_get_info()
    if free < 6 << 30:
        pytest.skip("needs 6 GB of device memory")
    big = torch.zeros(1 << 31, dtype=torch.bfloat16, device="cuda")
    try:
        numels = [4096 + 7, 1000, 333]
        dtypes = [torch.bfloat16, torch.float16, torch.float32]
        host, dev = make_list(numels, dtypes, seed=n_alias)
        base = torch.empty(numels[1] + 1, dtype=torch.float16, device="cuda")
        dev[1] = base[1:]
        dev[1].copy_(to_torch(host[1], torch.float16))
        dts = [TORCH_TO_DT[d] for d in dtypes]
        S = oracle.virtual_offsets([big.numel()] * n_alias + numels)[n_alias:]
        assert S[0] >= 1 << 36
        seed, eps = W.step_seed(n_alias), 1e-3
        plist = zo.ParamList([big] * n_alias + dev)
        theta = [bits_to_f64(storage_bits(h), dt).astype(np.float32) for h, dt in zip(host, dts)]
        for ops in (((5, -2 * eps),), ((5, eps), (6, eps)), ((7, eps), (8, eps))):
            if len(ops) == 1:
                zo.perturb(plist, seed, ops[0][0], ops[0][1])
            else:
                zo.perturb2(plist, seed, ops[0][0], ops[0][1], ops[1][0], ops[1][1])
            for i, (d, dt) in enumerate(zip(dev, dts)):
                g = np.uint64(S[i]) + np.arange(numels[i], dtype=np.uint64)
                for k, sc in ops:
                    want = oracle.perturb_elements(dt, g, theta[i], seed, k, sc)
                    theta[i] = bits_to_f64(want, dt).astype(np.float32)
                np.testing.assert_array_equal(storage_bits(d), want, err_msg=f"{n_alias} entries {ops} tensor {i}")
    finally:
        del big
        torch.cuda.empty_cache()


@pytest.mark.parametrize("n_alias", [32, 45])
@pytest.mark.parametrize("K,pre", [(16, True), (24, True), (40, False)])
def test_update_beyond_2_32_blocks(n_alias, K, pre):
    """Tensors whose Philox block counter has a non-zero high word (virtual
    index >= 2^36). One 2^31-element bf16 tensor (4 GB) listed n_alias times
    fills the index space below them. A launch holds fewer than 2^31 blocks
    (15 of these entries), so with 32 entries the checked tensors share a
    launch that starts below block 2^32 and ends above it (the general step);
    with 45 their launch starts above it (one high word for the whole launch:
    the split Philox of the 8-probe-table update). K = 16 takes the small-K
    kernel, 24 and 40 the chunked one with a last pair of one group. The
    aliased entries are updated concurrently and end with arbitrary values;
    only the checked tensors (bf16, a fp16 view off the 32-byte grid, fp32)
    are compared, element by element, with the oracle at their virtual
    indices."""
    free, _ = torch.cuda.mem_get_info()
    if free < 6 << 30:
        pytest.skip("needs 6 GB of device memory")
    big = torch.zeros(1 << 31, dtype=torch.bfloat16, device="cuda")
    try:
        numels = [4096 + 7, 1000, 333]
        dtypes = [torch.bfloat16, torch.float16, torch.float32]
        host, dev = make_list(numels, dtypes, seed=n_alias * 100 + K)
        base = torch.empty(numels[1] + 1, dtype=torch.float16, device="cuda")
        dev[1] = base[1:]
        dev[1].copy_(to_torch(host[1], torch.float16))
        dts = [TORCH_TO_DT[d] for d in dtypes]
        S = oracle.virtual_offsets([big.numel()] * n_alias + numels)[n_alias:]
        assert S[0] == n_alias << 31 and S[0] >= 1 << 36
        c_np = np.random.default_rng(K + n_alias).normal(0, 25, K)
        c = torch.tensor(c_np, dtype=torch.float64, device="cuda")
        seed, lr, eps = W.step_seed(K + n_alias), 1e-3, 1e-3
        zo.update([big] * n_alias + dev, seed, c, lr, pre=(K - 1, eps) if pre else None)
        for i, (d, h, dt) in enumerate(zip(dev, host, dts)):
            g = np.uint64(S[i]) + np.arange(h.size, dtype=np.uint64)
            theta = bits_to_f64(storage_bits(h), dt).astype(np.float32)
            if pre:
                theta = bits_to_f64(oracle.perturb_elements(dt, g, theta, seed, K - 1, eps), dt).astype(np.float32)
            want = oracle.update_elements(dt, g, theta, seed, c_np, lr)
            assert_update_close(storage_bits(d), want, dt, c_np, lr, context=f"{n_alias} entries K={K} tensor {i}")
    finally:
        del big
        torch.cuda.empty_cache()


def test_update_max_probes(packing_mode):
    K = zo.ZO_MAX_PROBES
    host, dev = make_list([5003, 16, 1], [torch.float32, torch.bfloat16, torch.float16], seed=77)
    dts = [W.DT_F32, W.DT_BF16, W.DT_F16]
    c_np = np.random.default_rng(77).normal(0, 5, K)
    c = torch.tensor(c_np, device="cuda")
    zo.update(dev, W.step_seed(77), c, 1e-2)
    oracle.update(host, dts, W.step_seed(77), c_np, 1e-2)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, 1e-2)
    with pytest.raises(zo.ZoError) as e:
        zo.update(dev, 1, torch.ones(K + 1, dtype=torch.float64, device="cuda"), 1e-3)
    assert e.value.status == zo.ZO_ERR_TOO_MANY_PROBES


@pytest.mark.parametrize("K", [1, 5, 16])
def test_update_sequential_bit_exact(K, packing_mode):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=50 + K)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    c_np = np.random.default_rng(K).normal(0, 25, K)
    c = torch.tensor(c_np, device="cuda")
    zo.update_sequential(dev, W.step_seed(K), c, 2e-3)
    oracle.update_sequential(host, dts, W.step_seed(K), c_np, 2e-3)
    assert_storage_equal(dev, host)


def test_update_K1_is_a_perturb_fp32():
    host, dev = make_list([70001], [torch.float32], seed=8)
    c = torch.tensor([3.25], dtype=torch.float64, device="cuda")
    d2 = [dev[0].clone()]
    zo.update(dev, W.step_seed(8), c, 1e-3)
    a0 = float(np.float32(-(1e-3 / 1) * 3.25))
    zo.perturb(d2, W.step_seed(8), 0, a0)
    assert torch.equal(dev[0], d2[0])


# ------------------------------------------------------------ precondition
def crafted_losses():
    rows = [[2.5, 2.5, 2.5], [2.5 + 1e-7, 2.5, 2.5], [3.04, 2.98, 3.0], [2.98, 2.96, 3.0],
            [50.0, 50.0, 0.0], [1.0, -1.0, 0.0], [0.0, 0.0, 1e-3]]
    return np.array(rows, dtype=np.float64)


@pytest.mark.parametrize("K", [1, 7, 16, 256, 1024])
@pytest.mark.parametrize("alpha,lam,one_sided,relative", [(0.1, 1.0, False, False), (0.0, 1.0, False, False),
                                                          (1.0, 1.0, False, False), (0.5, 3.0, False, False),
                                                          (0.1, 1.0, True, False), (0.1, 1.0, False, True),
                                                          (1.0, 1e-3, True, True)])
def test_precondition_vs_oracle(K, alpha, lam, one_sided, relative):
    L = W.synthetic_losses(K, step=K)
    cr = crafted_losses()
    L[: min(K, len(cr))] = cr[: min(K, len(cr))]
    eps = 1e-3
    Ld = torch.tensor(L, device="cuda")
    c, st, w, cv = zo.precondition(Ld, eps, alpha=alpha, lambda_reg=lam, one_sided=one_sided, relative=relative,
                                   with_weights=True)
    rc, c_o, w_o, cv_o = oracle.precondition(L, eps, alpha=alpha, lambda_reg=lam, one_sided=one_sided,
                                             relative=relative)
    assert rc == oracle.OK and int(st.item()) == zo.ZO_OK
    for got, want in ((c, c_o), (w, w_o), (cv, cv_o)):
        g = got.cpu().numpy()
        np.testing.assert_allclose(g, want, rtol=1e-6, atol=0)
        np.testing.assert_allclose(g, want, rtol=1e-13, atol=1e-300)


def test_precondition_relative_degenerate():
    """All-zero curvature (m = 0 -> w = 1/lambda_reg) and an overflowing mean."""
    eps = 1e-3
    L = np.array([[2.0, 2.0, 2.0], [2.5, 1.5, 2.0], [3.0, 1.0, 2.0]])
    c, st, w, _ = zo.precondition(torch.tensor(L, device="cuda"), eps, lambda_reg=0.5, relative=True,
                                  with_weights=True)
    rc, c_o, w_o, _ = oracle.precondition(L, eps, lambda_reg=0.5, relative=True)
    assert rc == oracle.OK and int(st.item()) == zo.ZO_OK
    np.testing.assert_array_equal(w.cpu().numpy(), w_o)
    np.testing.assert_allclose(c.cpu().numpy(), c_o, rtol=1e-15)
    big = 1.5e308 * 1e-6 / 2
    Lb = np.array([[big, big, 0.0], [big, big, 0.0]])
    sentinel = torch.full((2,), 7.0, dtype=torch.float64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    zo.precondition(torch.tensor(Lb, device="cuda"), eps, relative=True, out=(sentinel, status))
    assert int(status.item()) == zo.ZO_ERR_NONFINITE == oracle.precondition(Lb, eps, relative=True)[0]
    assert torch.all(sentinel == 7.0)


@pytest.mark.parametrize("bad", [np.nan, np.inf])
def test_precondition_nonfinite_blocks_update(bad):
    L = W.synthetic_losses(16, 0)
    L[5, 1] = bad
    Ld = torch.tensor(L, device="cuda")
    sentinel = torch.full((16,), 123.0, dtype=torch.float64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    c, st = zo.precondition(Ld, 1e-3, out=(sentinel, status))
    assert int(st.item()) == zo.ZO_ERR_NONFINITE
    assert torch.all(sentinel == 123.0)
    host, dev = make_list([1000], [torch.bfloat16])
    before = storage_np(dev[0])
    zo.update(dev, 1, c, 1e-3, status=st)
    zo.update_sequential(dev, 1, c, 1e-3, status=st)
    np.testing.assert_array_equal(storage_np(dev[0]), before)
    # a clean call resets the status and the update proceeds
    c2, st2 = zo.precondition(torch.tensor(W.synthetic_losses(16, 0), device="cuda"), 1e-3, out=(sentinel, status))
    assert int(st2.item()) == zo.ZO_OK
    zo.update(dev, 1, c2, 1e-3, status=st2)
    assert not np.array_equal(storage_np(dev[0]), before)


# --------------------------------------------------------------------- loss
@pytest.mark.parametrize("n", [0, 1, 1000, 1 << 20, (1 << 20) + 7, 3_000_001])
def test_quadratic_loss(n):
    th = W.tiny_theta(n) if n else np.zeros(0, np.float32)
    a = W.tiny_curvatures(n) if n else np.zeros(0, np.float32)
    td, ad = torch.from_numpy(th).cuda(), torch.from_numpy(a).cuda()
    got = zo.quadratic_loss(td, ad).item()
    want = oracle.quadratic_loss(th, a)
    assert got == pytest.approx(want, rel=1e-12, abs=0)
    assert zo.quadratic_loss(td, ad).item() == got   # fixed order: reproducible


def test_prepared_quadratic_loss():
    """QuadraticLoss (arguments checked once) writes the same value as
    quadratic_loss into any float64 cell, and rejects bad arguments."""
    n = (1 << 20) + 7
    td = torch.from_numpy(W.tiny_theta(n)).cuda()
    ad = torch.from_numpy(W.tiny_curvatures(n)).cuda()
    table = torch.full((4, 3), -1.0, dtype=torch.float64, device="cuda")
    q = zo.QuadraticLoss(td, ad)
    q(q.out_address(table[2, 1:2]))
    want = zo.quadratic_loss(td, ad).item()
    assert table[2, 1].item() == want
    assert (table.view(-1)[torch.arange(12, device="cuda") != 7] == -1.0).all()   # nothing else written
    with pytest.raises(ValueError):
        zo.QuadraticLoss(td, ad[:-1])
    with pytest.raises(ValueError):
        zo.QuadraticLoss(td, ad, workspace=torch.empty(8, dtype=torch.uint8, device="cuda"))
    with pytest.raises(ValueError):
        q.out_address(torch.empty(1, dtype=torch.float32, device="cuda"))
    with pytest.raises(TypeError):
        zo.QuadraticLoss(td, ad.double())


# ------------------------------------------------------- small workload, e2e
def test_tiny_workload_lockstep():
    """Ten full steps of the small workload (d = 2^20 fp32, quadratic loss,
    K = 8, eps = 1e-3, lr = 1e-2). Each step starts the oracle from the GPU's
    weights and compares every loss, coefficient and the updated weights."""
    ps = W.TINY
    th0, a = W.tiny_theta(), W.tiny_curvatures()
    theta = torch.from_numpy(th0).cuda()
    ad = torch.from_numpy(a).cuda()
    plist = zo.ParamList([theta])
    K, eps, lr = ps.K, ps.eps, W.TINY_LR
    losses = torch.empty(K, 3, dtype=torch.float64, device="cuda")
    ws = torch.empty(zo.quadratic_loss_workspace_size(theta.numel()), dtype=torch.uint8, device="cuda")
    for step in range(W.TINY_STEPS):
        seed = W.step_seed(step)
        host = [theta.cpu().numpy().copy()]
        # GPU step: the center loss first, once (Algorithm 1), then the probes
        l0 = zo.quadratic_loss(theta, ad, workspace=ws)
        for k in range(K):
            zo.perturb(plist, seed, k, eps)
            zo.quadratic_loss(theta, ad, out=losses[k, 0:1], workspace=ws)
            zo.perturb(plist, seed, k, -2 * eps)
            zo.quadratic_loss(theta, ad, out=losses[k, 1:2], workspace=ws)
            zo.perturb(plist, seed, k, eps)
        losses[:, 2] = l0
        c, st = zo.precondition(losses, eps)
        zo.update(plist, seed, c, lr, status=st)
        # oracle step from the same starting weights
        rows = []
        l0_o = oracle.quadratic_loss(host[0], a)
        for k in range(K):
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            lp = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
            lm = oracle.quadratic_loss(host[0], a)
            oracle.perturb(host, [W.DT_F32], seed, k, eps)
            rows.append([lp, lm, l0_o])
        rows = np.array(rows)
        Lg = losses.cpu().numpy()
        cg = c.cpu().numpy()
        assert int(st.item()) == zo.ZO_OK
        # losses: the same perturbed weights bit for bit; only the fp64
        # summation order differs
        np.testing.assert_allclose(Lg, rows, rtol=1e-12)
        # preconditioner on identical inputs
        rc, c_same, _, _ = oracle.precondition(Lg, eps)
        assert rc == oracle.OK
        np.testing.assert_allclose(cg, c_same, rtol=1e-12)
        # against the oracle's own losses: a relative loss error r becomes
        # r (|L+| + |L-|) / |L+ - L-| in the difference and
        # alpha r (|L+| + 2|L0| + |L-|) / |L+ - 2 L0 + L-| through w
        rc, c_o, _, _ = oracle.precondition(rows, eps)
        assert rc == oracle.OK
        lp, lm, l0 = np.abs(rows[:, 0]), np.abs(rows[:, 1]), np.abs(rows[:, 2])
        cond = ((lp + lm) / np.abs(rows[:, 0] - rows[:, 1])
                + 0.1 * (lp + 2 * l0 + lm) / np.abs(rows[:, 0] - 2 * rows[:, 2] + rows[:, 1]))
        assert np.all(np.abs(cg - c_o) <= 1e-11 * cond * np.abs(c_o) + 1e-300)
        oracle.update(host, [W.DT_F32], seed, cg, lr)
        assert_update_close(storage_bits(theta), storage_bits(host[0]), W.DT_F32, c.cpu().numpy(), lr,
                            context=f"step {step}")


# ------------------------------------------- fused passes of a step schedule
@pytest.mark.parametrize("a,b", [(3, 4), (7, 8), (5, 5), (0, 1023)])
def test_perturb2_is_two_perturbs(a, b, packing_mode):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=a + 31 * b)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    dev2 = [t.clone() for t in dev]
    seed, sa, sb = W.step_seed(a), 1e-3, -2.5e-3
    zo.perturb2(dev, seed, a, sa, b, sb)
    zo.perturb(dev2, seed, a, sa)
    zo.perturb(dev2, seed, b, sb)
    for x, y in zip(dev, dev2):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True
    oracle.perturb(host, dts, seed, a, sa)
    oracle.perturb(host, dts, seed, b, sb)
    assert_storage_equal(dev, host)


def test_perturb2_every_tuned_configuration():
    """zo_perturb2 times its three candidate configurations on the first nine
    calls for a parameter list with both probes in one group of 8 (three
    rounds), and on the first three with the probes in two groups (one
    round, a kernel of its own), then keeps the fastest of each: 12 calls of
    the first kind and 6 of the second on one list run every candidate and
    the chosen one, each bit-exact with the oracle."""
    rng = np.random.default_rng(606)
    numels = [int(x) for x in rng.integers(1, 70000, 40)] + [4096 * 300, 17]
    dtypes = [DTS[int(x)] for x in rng.integers(0, 3, len(numels))]
    host, dev = make_list(numels, dtypes, seed=606)
    dts = [TORCH_TO_DT[d] for d in dtypes]
    plist = zo.ParamList(dev)
    seed = W.step_seed(606)
    pairs = [(8 * c + 1, 8 * c + 2) for c in range(12)] + [(8 * c + 7, 8 * c + 8) for c in range(6)]
    for call, (a, b) in enumerate(pairs):
        zo.perturb2(plist, seed, a, 1e-3, b, -1e-3)
        oracle.perturb(host, dts, seed, a, 1e-3)
        oracle.perturb(host, dts, seed, b, -1e-3)
        torch.cuda.synchronize()
        assert_storage_equal(dev, host, f"call {call}")


def test_fused_step_in_a_cuda_graph():
    """Every call of a fused step only enqueues work on the current stream and
    allocates nothing, so a whole step can be captured into a CUDA graph and
    replayed (aligned tensors and views off the 32-byte grid): the replay
    matches the oracle's Algorithm 1 order."""
    K, eps = 4, 1e-3
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=808)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    rng = np.random.default_rng(809)
    for dtype, off, n in ((torch.bfloat16, 3, 5000), (torch.float32, 1, 777), (torch.float16, 5, 40)):
        h = W.random_storage(rng, n, TORCH_TO_DT[dtype])       # views off the 32-byte grid: the chunk kernels
        v = torch.empty(n + off, dtype=dtype, device="cuda")[off:]
        v.copy_(to_torch(h, dtype))
        host.append(h.copy())
        dev.append(v)
        dts.append(TORCH_TO_DT[dtype])

    def same_layout(t):
        off = (t.data_ptr() % 32) // t.element_size()
        return torch.empty(t.numel() + off, dtype=t.dtype, device="cuda")[off:].copy_(t)

    plist = zo.ParamList(dev)
    seed = W.step_seed(808)
    L = torch.tensor(W.synthetic_losses(K, 808), device="cuda")
    c = torch.empty(K, dtype=torch.float64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    scratch = zo.ParamList([same_layout(t) for t in dev])      # warm-up outside the capture
    zo.perturb(scratch, seed, 0, eps)
    zo.perturb2(scratch, seed, 0, eps, 1, eps)
    zo.precondition(L, eps, out=(c, st))
    zo.update(scratch, seed, c, eps, status=st, pre=(K - 1, eps))
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            zo.perturb(plist, seed, 0, eps)
            for k in range(K):
                zo.perturb(plist, seed, k, -2 * eps)
                if k + 1 < K:
                    zo.perturb2(plist, seed, k, eps, k + 1, eps)
            zo.precondition(L, eps, out=(c, st))
            zo.update(plist, seed, c, eps, status=st, pre=(K - 1, eps))
    torch.cuda.synchronize()
    assert_storage_equal(dev, host, "capture must not execute")
    g.replay()
    torch.cuda.synchronize()
    for k in range(K):
        for sc in (eps, -2 * eps, eps):
            oracle.perturb(host, dts, seed, k, sc)
    rc, c_o, _, _ = oracle.precondition(W.synthetic_losses(K, 808), eps)
    assert rc == oracle.OK and int(st.item()) == zo.ZO_OK
    np.testing.assert_allclose(c.cpu().numpy(), c_o, rtol=1e-12)
    oracle.update(host, dts, seed, c.cpu().numpy(), eps)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c.cpu().numpy(), eps, context="graph replay")


def test_concurrent_host_threads_on_their_own_streams():
    """Two host threads, each with its own parameter list and stream, call the
    library at the same time (the binding releases the GIL in every call):
    the per-thread launch state, the device table and the two-op tuner keep
    them apart, and each list matches the oracle."""
    import threading
    K, eps, iters = 6, 1e-3, 20
    jobs = []
    for j in range(2):
        numels = [4096 * 40 + 16 * j, 333, 70000 + j]
        dtypes = [torch.bfloat16, torch.float16, torch.float32]
        host, dev = make_list(numels, dtypes, seed=900 + j)
        jobs.append({"host": host, "dev": dev, "dts": [TORCH_TO_DT[d] for d in dtypes],
                     "seed": W.step_seed(900 + j), "stream": torch.cuda.Stream(), "err": None})

    def run(job):
        try:
            with torch.cuda.stream(job["stream"]):
                plist = zo.ParamList(job["dev"])
                seed = job["seed"]
                for it in range(iters):
                    zo.perturb(plist, seed, it, eps)
                    zo.perturb2(plist, seed, it, -eps, it + 1, 2 * eps)
                L = torch.tensor(W.synthetic_losses(K, 3), device="cuda")
                c, st = zo.precondition(L, eps)
                zo.update(plist, seed, c, eps, status=st, pre=(3, eps))
                job["c"] = c
            job["stream"].synchronize()
        except Exception as e:  # reported by the main thread
            job["err"] = e

    threads = [threading.Thread(target=run, args=(j,)) for j in jobs]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    for job in jobs:
        assert job["err"] is None, job["err"]
        host, dts, seed = job["host"], job["dts"], job["seed"]
        for it in range(iters):
            oracle.perturb(host, dts, seed, it, eps)
            oracle.perturb(host, dts, seed, it, -eps)
            oracle.perturb(host, dts, seed, it + 1, 2 * eps)
        oracle.perturb(host, dts, seed, 3, eps)
        c = job["c"].cpu().numpy()
        rc, c_o, _, _ = oracle.precondition(W.synthetic_losses(K, 3), eps)
        np.testing.assert_allclose(c, c_o, rtol=1e-12)
        oracle.update(host, dts, seed, c, eps)
        for d, h, dt in zip(job["dev"], host, dts):
            assert_update_close(storage_bits(d), storage_bits(h), dt, c, eps, context="concurrent threads")


@pytest.mark.parametrize("K", [1, 9, 64])
def test_update_with_leading_perturb(K, packing_mode):
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=K + 5)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    dev2 = [t.clone() for t in dev]
    c_np = np.random.default_rng(K).normal(0, 25, K)
    c = torch.tensor(c_np, device="cuda")
    seed, lr, eps = W.step_seed(K), 1e-3, 1e-3
    zo.update(dev, seed, c, lr, pre=(K - 1, eps))
    zo.perturb(dev2, seed, K - 1, eps)
    zo.update(dev2, seed, c, lr)
    for x, y in zip(dev, dev2):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True
    oracle.perturb(host, dts, seed, K - 1, eps)
    oracle.update(host, dts, seed, c_np, lr)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, lr)


@pytest.mark.parametrize("K,pre_probe", [(3, 1), (3, 9), (9, 3), (9, 40), (16, 100), (24, 200)])
def test_update_with_leading_perturb_of_another_probe(K, pre_probe, packing_mode):
    """The leading perturbation's probe in one of the update's own probe
    groups (its Philox word shared with the sums) or in another group (its own
    word), one or two groups: the same as the perturbation then the update."""
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=K + pre_probe)
    dts = [TORCH_TO_DT[d] for d in MIXED_DTYPES]
    dev2 = [t.clone() for t in dev]
    c_np = np.random.default_rng(K + pre_probe).normal(0, 25, K)
    c = torch.tensor(c_np, device="cuda")
    seed, lr, eps = W.step_seed(pre_probe), 1e-3, -2e-3
    zo.update(dev, seed, c, lr, pre=(pre_probe, eps))
    zo.perturb(dev2, seed, pre_probe, eps)
    zo.update(dev2, seed, c, lr)
    for x, y in zip(dev, dev2):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True
    oracle.perturb(host, dts, seed, pre_probe, eps)
    oracle.update(host, dts, seed, c_np, lr)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, lr)


def test_update_with_leading_perturb_after_failed_preconditioner():
    """A non-finite loss skips the probe sum but never the restore."""
    host, dev = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=99)
    dev2 = [t.clone() for t in dev]
    L = W.synthetic_losses(8, 0)
    L[2, 0] = np.nan
    c, st = zo.precondition(torch.tensor(L, device="cuda"), 1e-3)
    assert int(st.item()) == zo.ZO_ERR_NONFINITE
    zo.update(dev, 3, c, 1e-3, status=st, pre=(7, 1e-3))
    zo.perturb(dev2, 3, 7, 1e-3)
    for x, y in zip(dev, dev2):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True


def test_fused_schedule_matches_algorithm1(packing_mode):
    """A whole step with restores folded into the next probe's +eps and into
    the update gives, bit for bit, the weights Algorithm 1's schedule gives at
    every point a forward pass would see them, and at the end."""
    K, eps, lr = 6, 1e-3, 1e-3
    _, dev_a = make_list(MIXED_NUMELS, MIXED_DTYPES, seed=123)
    dev_b = [t.clone() for t in dev_a]
    seed = W.step_seed(42)
    L = torch.tensor(W.synthetic_losses(K, 42), device="cuda")
    c, st = zo.precondition(L, eps)

    def snap(ts):
        return [t.clone() for t in ts]

    seen_a, seen_b = [], []
    for k in range(K):                         # Algorithm 1
        zo.perturb(dev_a, seed, k, eps)
        seen_a.append(snap(dev_a))
        zo.perturb(dev_a, seed, k, -2 * eps)
        seen_a.append(snap(dev_a))
        zo.perturb(dev_a, seed, k, eps)
    zo.update(dev_a, seed, c, lr, status=st)
    zo.perturb(dev_b, seed, 0, eps)            # fused schedule: 2K + 1 passes
    for k in range(K):
        seen_b.append(snap(dev_b))
        zo.perturb(dev_b, seed, k, -2 * eps)
        seen_b.append(snap(dev_b))
        if k + 1 < K:
            zo.perturb2(dev_b, seed, k, eps, k + 1, eps)
    zo.update(dev_b, seed, c, lr, status=st, pre=(K - 1, eps))
    for sa, sb in zip(seen_a + [dev_a], seen_b + [dev_b]):
        for x, y in zip(sa, sb):
            assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True


def test_fused_calls_on_split_launches_and_unaligned_views(packing_mode):
    """zo_perturb2 and zo_update_ex on 2500 tensors of odd sizes and mixed
    dtypes (several launches) plus unaligned views (aligned-chunk path): bit
    for bit the unfused calls."""
    rng = np.random.default_rng(77)
    numels = [int(x) for x in rng.integers(0, 200, 2500)]
    dtypes = [DTS[int(x)] for x in rng.integers(0, 3, 2500)]
    _, dev = make_list(numels, dtypes, seed=77)
    base = torch.randn(5000, device="cuda").to(torch.bfloat16)
    dev += [base[1:1 + 777], base[1000 + 3:1000 + 3 + 2049]]      # 2-byte aligned views
    dev2 = [t.clone() for t in dev]
    seed, eps = W.step_seed(77), 1e-3
    c = torch.tensor(rng.normal(0, 20, 11), dtype=torch.float64, device="cuda")
    zo.perturb2(dev, seed, 7, eps, 8, -eps)
    zo.update(dev, seed, c, 1e-3, pre=(10, eps))
    zo.perturb(dev2, seed, 7, eps)
    zo.perturb(dev2, seed, 8, -eps)
    zo.perturb(dev2, seed, 10, eps)
    zo.update(dev2, seed, c, 1e-3)
    for x, y in zip(dev, dev2):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)) if x.numel() else True


def test_binding_rejects_bad_output_buffers():
    """The binding checks what the library will write: the coefficient and
    status buffers' sizes and dtypes, the loss output's dtype."""
    L = torch.tensor(W.synthetic_losses(8, 0), device="cuda")
    with pytest.raises(ValueError):
        zo.precondition(L, 1e-3, out=(torch.empty(7, dtype=torch.float64, device="cuda"),
                                      torch.empty(1, dtype=torch.int32, device="cuda")))
    with pytest.raises(TypeError):
        zo.precondition(L, 1e-3, out=(torch.empty(8, dtype=torch.float32, device="cuda"),
                                      torch.empty(1, dtype=torch.int32, device="cuda")))
    th = torch.zeros(100, device="cuda")
    with pytest.raises(TypeError):
        zo.quadratic_loss(th, th, out=torch.empty(1, dtype=torch.float32, device="cuda"))
    with pytest.raises(ValueError):
        zo.quadratic_loss_static(th, th, out=torch.empty(0, dtype=torch.float64, device="cuda"))
    with pytest.raises(TypeError):
        zo.update([th], 1, torch.zeros(4, dtype=torch.float32, device="cuda"), 1e-3)
