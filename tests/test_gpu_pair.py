"""GPU parity of zo_perturb_pair (both forward points of a probe, out of
place) against the CPU oracle: plus and minus must equal the oracle's
perturbation of a copy of theta by +scale and -scale, bit for bit, and theta
must stay untouched. Also the schedule built on it: K pair passes, the
preconditioner and the fused update leave theta where the oracle's update of
the unperturbed theta puts it."""
import gc

import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

from gpu_helpers import (TORCH_TO_DT, assert_update_close, gather, sample_positions, storage_bits, storage_np,
                         to_torch)

pytestmark = pytest.mark.gpu

DTS = [torch.float32, torch.bfloat16, torch.float16]
NUMELS = [1, 15, 16, 17, 31, 33, 0, 255, 4096, 4099, 100003, 7, 65536 + 5]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def make(numels, dtypes, seed):
    rng = np.random.default_rng(seed)
    host = [W.random_storage(rng, n, TORCH_TO_DT[dt]) for n, dt in zip(numels, dtypes)]
    return host, [to_torch(h, dt) for h, dt in zip(host, dtypes)]


def like(dev, fill_seed):
    """Buffers shaped like dev, filled with unrelated bits (the kernel must
    overwrite every element)."""
    g = torch.Generator(device="cuda").manual_seed(fill_seed)
    out = []
    for t in dev:
        b = torch.empty_like(t)
        if b.numel():
            b.view(torch.uint8).copy_(torch.randint(0, 256, (b.numel() * b.element_size(),), generator=g,
                                                    device="cuda", dtype=torch.uint8))
        out.append(b)
    return out


def expect(host, dts, seed, k, scale):
    plus = [h.copy() for h in host]
    minus = [h.copy() for h in host]
    oracle.perturb(plus, dts, seed, k, scale)
    oracle.perturb(minus, dts, seed, k, -scale)
    return plus, minus


def assert_equal(dev, host, what):
    for i, (d, h) in enumerate(zip(dev, host)):
        got = storage_np(d)
        view = np.uint32 if h.dtype == np.float32 else np.uint16
        np.testing.assert_array_equal(got.view(view), h.view(view), err_msg=f"{what} tensor {i} numel {h.size}")


@pytest.mark.parametrize("k,scale", [(0, 1e-3), (9, 1e-3), (255, 0.25), (1023, -3e-8)])
def test_pair_bit_exact_mixed(k, scale, packing_mode):
    dtypes = [DTS[i % 3] for i in range(len(NUMELS))]
    dts = [TORCH_TO_DT[d] for d in dtypes]
    host, dev = make(NUMELS, dtypes, seed=k)
    plus, minus = like(dev, 1), like(dev, 2)
    seed = W.step_seed(4)
    zo.perturb_pair(dev, plus, minus, seed, k, scale)
    want_p, want_m = expect(host, dts, seed, k, scale)
    assert_equal(plus, want_p, "plus")
    assert_equal(minus, want_m, "minus")
    assert_equal(dev, host, "theta untouched")


@pytest.mark.parametrize("which", ["theta", "plus", "minus"])
@pytest.mark.parametrize("offset", [1, 8, 16])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float16, torch.float32])
def test_pair_unaligned(which, offset, dtype):
    """One of the three pointers off the 32-byte grid, the others aligned:
    theta -> the aligned-chunk kernel with theta read from its segments;
    plus or minus -> the per-block path with the widest accesses each
    address allows. Results are identical and nothing outside the views is
    written."""
    n = 4096 + 37
    dt = TORCH_TO_DT[dtype]
    rng = np.random.default_rng(offset)
    bases = {}
    views = {}
    for name in ("theta", "plus", "minus"):
        off = offset if name == which else 0
        h = W.random_storage(rng, n + off + 64, dt)
        bases[name] = (h, to_torch(h, dtype), off)
        views[name] = bases[name][1][off:off + n]
    host = [bases["theta"][0][bases["theta"][2]:bases["theta"][2] + n].copy()]
    seed = W.step_seed(7)
    zo.perturb_pair([views["theta"]], [views["plus"]], [views["minus"]], seed, 21, 1e-3)
    want_p, want_m = expect(host, [dt], seed, 21, 1e-3)
    assert_equal([views["plus"]], want_p, "plus")
    assert_equal([views["minus"]], want_m, "minus")
    for name in ("plus", "minus", "theta"):
        h, d, off = bases[name]
        after = storage_np(d)
        np.testing.assert_array_equal(after[:off], h[:off])
        np.testing.assert_array_equal(after[off + n:], h[off + n:])


@pytest.mark.parametrize("dtype", DTS)
def test_pair_every_shared_offset(dtype, packing_mode):
    """theta, plus and minus all views at the same element offset (every
    offset off the 32-byte grid; fp32 also at offset 0): the aligned-chunk
    pair kernel, bit for bit the oracle, nothing outside the views written."""
    per = 32 // torch.tensor([], dtype=dtype).element_size()
    offsets = list(range(1, per)) + ([0] if dtype == torch.float32 else [])
    sizes = [1, 3, 15, 16, 17, 100, 4096 + 37, 20011]
    dt = TORCH_TO_DT[dtype]
    rng = np.random.default_rng(per)
    theta, plus, minus, host, guards = [], [], [], [], []
    for i, off in enumerate(offsets):
        n = sizes[i % len(sizes)]
        for lst in (theta, plus, minus):
            h = W.random_storage(rng, off + n + 40, dt)
            b = to_torch(h, dtype)
            guards.append((h, b, off, n))
            lst.append(b[off:off + n])
        host.append(storage_np(theta[-1]).copy())
    seed = W.step_seed(12)
    zo.perturb_pair(theta, plus, minus, seed, 29, 1e-3)
    want_p, want_m = expect(host, [dt] * len(host), seed, 29, 1e-3)
    assert_equal(plus, want_p, "plus")
    assert_equal(minus, want_m, "minus")
    assert_equal(theta, host, "theta untouched")
    for h, b, off, n in guards[0::3]:                   # theta's allocations: untouched entirely
        np.testing.assert_array_equal(storage_np(b), h)
    for h, b, off, n in guards[1::3] + guards[2::3]:    # outputs: nothing outside the views
        after = storage_np(b)
        np.testing.assert_array_equal(after[:off], h[:off])
        np.testing.assert_array_equal(after[off + n:], h[off + n:])


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float16])
@pytest.mark.parametrize("out_off", [0, 5])
def test_pair_theta_at_another_offset(dtype, out_off, packing_mode):
    """theta at every element offset, plus and minus sharing another one (0:
    fresh allocations): chunks follow the outputs and theta is read from the
    aligned segments that hold each chunk's elements; bit for bit the oracle,
    nothing outside the views written."""
    sizes = [1, 3, 15, 16, 17, 100, 4096 + 37, 20011]
    dt = TORCH_TO_DT[dtype]
    rng = np.random.default_rng(60 + out_off)
    theta, plus, minus, host, guards = [], [], [], [], []
    for i, off in enumerate(o for o in range(16) if o != out_off):
        n = sizes[i % len(sizes)]
        for lst, o in ((theta, off), (plus, out_off), (minus, out_off)):
            h = W.random_storage(rng, o + n + 40, dt)
            b = to_torch(h, dtype)
            guards.append((h, b, o, n))
            lst.append(b[o:o + n])
        host.append(storage_np(theta[-1]).copy())
    seed = W.step_seed(14)
    zo.perturb_pair(theta, plus, minus, seed, 30, -1e-3)
    want_p, want_m = expect(host, [dt] * len(host), seed, 30, -1e-3)
    assert_equal(plus, want_p, "plus")
    assert_equal(minus, want_m, "minus")
    for h, b, off, n in guards[0::3]:
        np.testing.assert_array_equal(storage_np(b), h)
    for h, b, off, n in guards[1::3] + guards[2::3]:
        after = storage_np(b)
        np.testing.assert_array_equal(after[:off], h[:off])
        np.testing.assert_array_equal(after[off + n:], h[off + n:])


def test_pair_many_fp32_tensors(packing_mode):
    """More fp32 tensors in one launch than one chunk-kernel launch takes
    (512): the host splits them."""
    rng = np.random.default_rng(41)
    numels = [int(x) for x in rng.integers(0, 90, 1000)]
    host, dev = make(numels, [torch.float32] * len(numels), seed=41)
    plus, minus = like(dev, 11), like(dev, 12)
    seed = W.step_seed(13)
    zo.perturb_pair(dev, plus, minus, seed, 5, 2e-3)
    want_p, want_m = expect(host, [W.DT_F32] * len(host), seed, 5, 2e-3)
    assert_equal(plus, want_p, "plus")
    assert_equal(minus, want_m, "minus")


def test_pair_split_launches(packing_mode):
    """More tensors than one launch holds (1024)."""
    rng = np.random.default_rng(31)
    numels = [int(x) for x in rng.integers(0, 300, 2300)]
    dtypes = [DTS[int(x)] for x in rng.integers(0, 3, 2300)]
    dts = [TORCH_TO_DT[d] for d in dtypes]
    host, dev = make(numels, dtypes, seed=31)
    plus, minus = like(dev, 3), like(dev, 4)
    seed = W.step_seed(8)
    zo.perturb_pair(dev, plus, minus, seed, 77, 2e-3)
    want_p, want_m = expect(host, dts, seed, 77, 2e-3)
    assert_equal(plus, want_p, "plus")
    assert_equal(minus, want_m, "minus")


def test_pair_matches_in_place_perturb():
    """plus equals zo_perturb(+scale) of a copy and minus zo_perturb(-scale),
    on the GPU, bit for bit; plus may alias theta."""
    dtypes = [DTS[i % 3] for i in range(len(NUMELS))]
    _, dev = make(NUMELS, dtypes, seed=5)
    a = [t.clone() for t in dev]
    b = [t.clone() for t in dev]
    seed = W.step_seed(2)
    zo.perturb(a, seed, 14, 1e-3)
    zo.perturb(b, seed, 14, -1e-3)
    minus = like(dev, 6)
    zo.perturb_pair(dev, dev, minus, seed, 14, 1e-3)      # plus aliases theta
    assert_equal(dev, [storage_np(t) for t in a], "plus (aliasing theta) vs zo_perturb(+scale)")
    assert_equal(minus, [storage_np(t) for t in b], "minus vs zo_perturb(-scale)")


def test_pair_rejects_same_plus_and_minus():
    _, dev = make([64], [torch.bfloat16], seed=1)
    buf = like(dev, 7)
    with pytest.raises(zo.ZoError):
        zo.perturb_pair(dev, buf, buf, 1, 0, 1e-3)


@pytest.mark.parametrize("K", [8, 19])
def test_pair_schedule_step(K, packing_mode):
    """K pair passes (theta untouched), the preconditioner, the fused update:
    theta ends where the oracle's update of the unperturbed theta puts it, and
    every pair matched the oracle's theta +- eps z_k."""
    dtypes = [torch.bfloat16, torch.float16, torch.float32, torch.bfloat16]
    numels = [5000, 4096 * 3 + 5, 777, 65536]
    dts = [TORCH_TO_DT[d] for d in dtypes]
    host, dev = make(numels, dtypes, seed=K)
    plus, minus = like(dev, 8), like(dev, 9)
    seed, eps = W.step_seed(K), 1e-3
    for k in range(K):
        zo.perturb_pair(dev, plus, minus, seed, k, eps)
        if k in (0, K - 1):
            want_p, want_m = expect(host, dts, seed, k, eps)
            assert_equal(plus, want_p, f"plus k={k}")
            assert_equal(minus, want_m, f"minus k={k}")
    assert_equal(dev, host, "theta untouched by the pair passes")
    L = W.synthetic_losses(K, step=K)
    c, st = zo.precondition(torch.tensor(L, device="cuda"), eps)
    zo.update(dev, seed, c, eps, status=st)
    c_h = c.cpu().numpy()
    oracle.update(host, dts, seed, c_h, eps)
    for d, h, dt in zip(dev, host, dts):
        assert_update_close(storage_bits(d), storage_bits(h), dt, c_h, eps, context="pair schedule")


@pytest.mark.parametrize("key", ["opt-13b", "opt-30b"])
def test_pair_fullsize_sampled(key):
    """Full-size sets with three copies on the device (77 GB, 180 GB): sampled
    elements of plus and minus against the oracle, theta untouched."""
    ps = W.BY_KEY[key]
    free, _ = torch.cuda.mem_get_info()
    if free < 3 * ps.d * ps.bytes_per_elem * 1.05:
        pytest.skip(f"needs three copies of the {key}-shaped set")
    params = W.allocate_params(ps)
    plus = [torch.empty_like(t) for t in params]
    minus = [torch.empty_like(t) for t in params]
    try:
        S = oracle.virtual_offsets(ps.numels)
        t_idx, i_idx = sample_positions(ps.numels)
        g = (S[t_idx] + i_idx).astype(np.uint64)
        seed, k = W.step_seed(1), ps.K - 1
        bits0, f0 = gather(params, t_idx, i_idx)
        zo.perturb_pair(zo.ParamList(params), zo.ParamList(plus), zo.ParamList(minus), seed, k, ps.eps)
        bp, _ = gather(plus, t_idx, i_idx)
        bm, _ = gather(minus, t_idx, i_idx)
        np.testing.assert_array_equal(bp, oracle.perturb_elements(ps.dtype, g, f0, seed, k, ps.eps))
        np.testing.assert_array_equal(bm, oracle.perturb_elements(ps.dtype, g, f0, seed, k, -ps.eps))
        np.testing.assert_array_equal(gather(params, t_idx, i_idx)[0], bits0)   # theta untouched
    finally:
        del params, plus, minus
        gc.collect()
        torch.cuda.empty_cache()
