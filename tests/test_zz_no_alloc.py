"""zo_quadratic_loss_static -- the allocation-free quadratic loss -- against
the workspace version zo_quadratic_loss, both called through the C ABI.

The static variant serves callers that cannot allocate device memory: code
running inside a device-memory budget fixed in advance (a framework whose
caching allocator already holds the memory, where one more cudaMalloc fails)
or code that must not let an allocation synchronise the device. It keeps its
scratch in a fixed array compiled into the library, so every call shares that
array and keeps the previous call's contents.

This file is collected last: if it fails, a run that stops at the first
failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import workloads as W
from paper_2609_38095_gb300 import zo

pytestmark = pytest.mark.gpu

MAX_N = zo.ZO_QUADRATIC_LOSS_STATIC_MAX_N


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    zo_build.build()


def inputs(n):
    if n == 0:
        return torch.zeros(0, device="cuda"), torch.zeros(0, device="cuda")
    return torch.from_numpy(W.tiny_theta(n)).cuda(), torch.from_numpy(W.tiny_curvatures(n)).cuda()


def call_static(theta, a, out):
    """One call of the new entry point through the C ABI, into a caller buffer."""
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return zo._lib().zo_quadratic_loss_static(ctypes.c_void_p(theta.data_ptr()), ctypes.c_void_p(a.data_ptr()),
                                              theta.numel(), ctypes.c_void_p(out.data_ptr()), stream)


@pytest.mark.parametrize("n", [1 << 20, 3_000_001, MAX_N, 1, 0])
def test_static_matches_workspace_version_twice(n):
    theta, a = inputs(n)
    want = zo.quadratic_loss(theta, a).item()          # existing entry point (caller workspace)
    out = torch.full((2,), float("nan"), dtype=torch.float64, device="cuda")
    assert call_static(theta, a, out[0:1]) == zo.ZO_OK
    assert call_static(theta, a, out[1:2]) == zo.ZO_OK
    got = out.cpu().numpy()
    for v in got:
        assert v == pytest.approx(want, rel=1e-12, abs=0)  # the loss tolerance used throughout the tests
    assert got[0] == got[1]


def test_static_after_a_larger_call():
    """The shared array keeps the previous call's partial sums; a smaller call
    right after a larger one must not pick any of them up."""
    big_t, big_a = inputs(MAX_N)
    small_t, small_a = inputs(5000)
    out = torch.empty(3, dtype=torch.float64, device="cuda")
    assert call_static(big_t, big_a, out[0:1]) == zo.ZO_OK
    assert call_static(small_t, small_a, out[1:2]) == zo.ZO_OK
    assert call_static(big_t, big_a, out[2:3]) == zo.ZO_OK
    got = out.cpu().numpy()
    assert got[0] == pytest.approx(zo.quadratic_loss(big_t, big_a).item(), rel=1e-12, abs=0)
    assert got[1] == pytest.approx(zo.quadratic_loss(small_t, small_a).item(), rel=1e-12, abs=0)
    assert got[2] == got[0]


def test_static_rejects_beyond_capacity():
    theta, a = inputs(16)
    out = torch.full((1,), 7.0, dtype=torch.float64, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = zo._lib().zo_quadratic_loss_static(ctypes.c_void_p(theta.data_ptr()), ctypes.c_void_p(a.data_ptr()),
                                            MAX_N + 1, ctypes.c_void_p(out.data_ptr()), stream)
    assert rc == zo.ZO_ERR_WORKSPACE
    assert out.item() == 7.0   # nothing enqueued
    with pytest.raises(zo.ZoError):
        zo._check("zo_quadratic_loss_static", rc)
