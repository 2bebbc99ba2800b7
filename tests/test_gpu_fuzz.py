"""Seeded fuzzing of the parameter-list handling: random lists (empty, tiny,
odd-sized and large tensors, all three dtypes, views at random element
offsets, so every alignment class) driven through random sequences of
zo_perturb, zo_perturb2 (every tuned configuration: each list starts with ten
two-op calls), zo_perturb_pair and zo_update_ex, each result checked
against the oracle: bit-exact for the perturbations, within the derived
tolerance for the update."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

from gpu_helpers import TORCH_TO_DT, assert_update_close, storage_bits, storage_np, to_torch

pytestmark = pytest.mark.gpu

DTS = [torch.float32, torch.bfloat16, torch.float16]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()
    oracle.lib()


def random_list(rng):
    n = int(rng.integers(1, 40))
    host, dev, keep = [], [], []
    for _ in range(n):
        kind = rng.random()
        if kind < 0.15:
            numel = 0
        elif kind < 0.45:
            numel = int(rng.integers(1, 48))
        elif kind < 0.9:
            numel = int(rng.integers(48, 6000))
        else:
            numel = int(rng.integers(6000, 100000))
        dtype = DTS[int(rng.integers(0, 3))]
        dt = TORCH_TO_DT[dtype]
        off = int(rng.integers(0, 20)) if rng.random() < 0.4 else 0
        base_host = W.random_storage(rng, numel + off + 8, dt)
        base = to_torch(base_host, dtype)
        keep.append(base)
        dev.append(base[off:off + numel])
        host.append(base_host[off:off + numel].copy())
    return host, dev, keep


def assert_same(dev, host, what):
    for i, (d, h) in enumerate(zip(dev, host)):
        view = np.uint32 if h.dtype == np.float32 else np.uint16
        np.testing.assert_array_equal(storage_np(d).view(view), h.view(view), err_msg=f"{what}: tensor {i}")


@pytest.mark.parametrize("case", range(40))
def test_fuzz_lists_and_sequences(case):
    rng = np.random.default_rng(5000 + case)
    host, dev, keep = random_list(rng)
    dts = [TORCH_TO_DT[t.dtype] for t in dev]
    plist = zo.ParamList(dev)
    seed = W.step_seed(int(rng.integers(0, 2**32)))
    packing = int(rng.choice([1, 8]))
    with oracle.packing(packing), zo.packing(packing):
        for step in range(22):
            op = 0.5 if step < 10 else rng.random()   # ten two-op calls first: every tuned configuration
            k = int(rng.integers(0, 1024))
            scale = float(rng.choice([1e-3, -2e-3, 0.25, -3e-7]))
            if op < 0.25:
                zo.perturb(plist, seed, k, scale)
                oracle.perturb(host, dts, seed, k, scale)
                assert_same(dev, host, f"step {step} perturb")
            elif op < 0.7:
                k2 = int(rng.integers(0, 1024))
                s2 = float(rng.choice([1e-3, -1e-3, 2e-3]))
                zo.perturb2(plist, seed, k, scale, k2, s2)
                oracle.perturb(host, dts, seed, k, scale)
                oracle.perturb(host, dts, seed, k2, s2)
                assert_same(dev, host, f"step {step} perturb2")
            elif op < 0.85:
                plus = [torch.empty_like(t) for t in dev]
                minus = [torch.empty_like(t) for t in dev]
                zo.perturb_pair(plist, plus, minus, seed, k, scale)
                hp, hm = [h.copy() for h in host], [h.copy() for h in host]
                oracle.perturb(hp, dts, seed, k, scale)
                oracle.perturb(hm, dts, seed, k, -scale)
                assert_same(plus, hp, f"step {step} pair plus")
                assert_same(minus, hm, f"step {step} pair minus")
                assert_same(dev, host, f"step {step} pair theta")
            else:
                K = int(rng.integers(1, 40))
                c_np = rng.normal(0, 20, K)
                pre = (int(rng.integers(0, K)), 1e-3) if rng.random() < 0.5 else None
                zo.update(plist, seed, torch.tensor(c_np, device="cuda"), 1e-3, pre=pre)
                if pre is not None:
                    oracle.perturb(host, dts, seed, pre[0], pre[1])
                oracle.update(host, dts, seed, c_np, 1e-3)
                for i, (d, h, dt) in enumerate(zip(dev, host, dts)):
                    assert_update_close(storage_bits(d), storage_bits(h), dt, c_np, 1e-3,
                                        context=f"case {case} step {step} tensor {i}")
                # continue bit-exact from the GPU's state
                host = [storage_np(d).copy() for d in dev]
    torch.cuda.synchronize()
    del keep
