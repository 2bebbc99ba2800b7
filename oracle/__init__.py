"""CPU oracle for the 1.5-SPSA parameter-space step (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. It shares no code with the CUDA library
in ``paper_2609_38095_gb300`` and never imports it.

This module only marshals numpy arrays into ``zo_oracle.c``; every piece of the
method's arithmetic lives in that C file, where each routine cites the passage
of the paper it follows.
"""
import ctypes
import os

import numpy as np

from . import build as _build

F32, BF16, F16 = 0, 1, 2
OK, ERR_ARG, ERR_NONFINITE = 0, -1, -4

_lib = None
_u64p = ctypes.POINTER(ctypes.c_uint64)


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        c = ctypes
        L.oracle_philox4x32_10.argtypes = [c.c_void_p, c.c_void_p, c.c_void_p]
        L.oracle_probe_bit.argtypes = [c.c_uint64, c.c_uint32, c.c_uint64]
        L.oracle_probe_bit.restype = c.c_int
        L.oracle_probe_sign.argtypes = [c.c_uint64, c.c_uint32, c.c_uint64]
        L.oracle_probe_sign.restype = c.c_int
        L.oracle_probe_bytes.argtypes = [c.c_uint64, c.c_uint32, c.c_int64, c.c_int64, c.c_void_p]
        L.oracle_probe_signs.argtypes = [c.c_uint64, c.c_uint32, c.c_int64, c.c_int64, c.c_void_p]
        L.oracle_virtual_offsets.argtypes = [c.c_int32, c.c_void_p, c.c_void_p]
        L.oracle_bf16_to_f32.argtypes = [c.c_uint16]
        L.oracle_bf16_to_f32.restype = c.c_float
        L.oracle_f32_to_bf16.argtypes = [c.c_float]
        L.oracle_f32_to_bf16.restype = c.c_uint16
        L.oracle_f16_to_f32.argtypes = [c.c_uint16]
        L.oracle_f16_to_f32.restype = c.c_float
        L.oracle_f32_to_f16.argtypes = [c.c_float]
        L.oracle_f32_to_f16.restype = c.c_uint16
        tens = [c.c_int32, c.c_void_p, c.c_void_p, c.c_void_p]
        L.oracle_perturb.argtypes = tens + [c.c_uint64, c.c_uint32, c.c_float]
        L.oracle_perturb.restype = c.c_int
        L.oracle_perturb_elements.argtypes = [c.c_int32, c.c_int64, c.c_void_p, c.c_void_p, c.c_uint64,
                                              c.c_uint32, c.c_float, c.c_void_p]
        L.oracle_perturb_elements.restype = c.c_int
        L.oracle_precondition.argtypes = [c.c_void_p, c.c_int32, c.c_double, c.c_double, c.c_double,
                                          c.c_int32, c.c_void_p, c.c_void_p, c.c_void_p]
        L.oracle_precondition.restype = c.c_int
        L.oracle_update.argtypes = tens + [c.c_uint64, c.c_void_p, c.c_int32, c.c_double]
        L.oracle_update.restype = c.c_int
        L.oracle_update_sequential.argtypes = tens + [c.c_uint64, c.c_void_p, c.c_int32, c.c_double]
        L.oracle_update_sequential.restype = c.c_int
        L.oracle_update_elements.argtypes = [c.c_int32, c.c_int64, c.c_void_p, c.c_void_p, c.c_uint64,
                                             c.c_void_p, c.c_int32, c.c_double, c.c_void_p]
        L.oracle_update_elements.restype = c.c_int
        L.oracle_quadratic_loss.argtypes = [c.c_void_p, c.c_void_p, c.c_int64]
        L.oracle_quadratic_loss.restype = c.c_double
        _lib = L
    return _lib


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


# ----------------------------------------------------------------- generator
def philox4x32_10(ctr, key):
    """Raw Philox4x32-10 block: ctr is 4 uint32, key is 2 uint32."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def probe_bit(seed, k, g):
    return lib().oracle_probe_bit(seed, k, g)


def probe_sign(seed, k, g):
    return lib().oracle_probe_sign(seed, k, g)


def probe_bytes(seed, k, first, n):
    out = np.zeros(n, dtype=np.uint8)
    lib().oracle_probe_bytes(seed, k, first, n, _ptr(out))
    return out


def probe_signs(seed, k, first, n):
    out = np.zeros(n, dtype=np.int8)
    lib().oracle_probe_signs(seed, k, first, n, _ptr(out))
    return out


def virtual_offsets(numels):
    n = np.ascontiguousarray(numels, dtype=np.int64)
    out = np.zeros(len(n), dtype=np.int64)
    lib().oracle_virtual_offsets(len(n), _ptr(n), _ptr(out))
    return out


# ---------------------------------------------------------- storage formats
def f32_to_bf16(x):
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    return np.array([lib().oracle_f32_to_bf16(float(v)) for v in x], dtype=np.uint16)


def bf16_to_f32(h):
    h = np.ascontiguousarray(h, dtype=np.uint16).ravel()
    return np.array([lib().oracle_bf16_to_f32(int(v)) for v in h], dtype=np.float32)


def f32_to_f16(x):
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    return np.array([lib().oracle_f32_to_f16(float(v)) for v in x], dtype=np.uint16)


def f16_to_f32(h):
    h = np.ascontiguousarray(h, dtype=np.uint16).ravel()
    return np.array([lib().oracle_f16_to_f32(int(v)) for v in h], dtype=np.float32)


# ------------------------------------------------------------- tensor lists
def _table(tensors, dtypes):
    """tensors: list of numpy arrays holding raw storage (float32 or uint16)."""
    n = len(tensors)
    for t in tensors:
        assert t.flags["C_CONTIGUOUS"] and t.flags["WRITEABLE"]
    ptrs = (ctypes.c_void_p * max(n, 1))(*[t.ctypes.data for t in tensors])
    numel = np.array([t.size for t in tensors], dtype=np.int64)
    dt = np.array(dtypes, dtype=np.int32)
    return n, ptrs, numel, dt


def perturb(tensors, dtypes, seed, k, scale):
    """In place on the numpy storage arrays."""
    n, ptrs, numel, dt = _table(tensors, dtypes)
    rc = lib().oracle_perturb(n, ptrs, _ptr(numel), _ptr(dt), seed, k, ctypes.c_float(scale))
    if rc != OK:
        raise RuntimeError(f"oracle_perturb: {rc}")


def perturb_elements(dtype, g, theta, seed, k, scale):
    g = np.ascontiguousarray(g, dtype=np.uint64)
    th = np.ascontiguousarray(theta, dtype=np.float32)
    out = np.zeros(len(g), dtype=np.uint32)
    rc = lib().oracle_perturb_elements(dtype, len(g), _ptr(g), _ptr(th), seed, k, ctypes.c_float(scale), _ptr(out))
    if rc != OK:
        raise RuntimeError(f"oracle_perturb_elements: {rc}")
    return out


def precondition(losses, eps, alpha=0.1, lambda_reg=1.0, one_sided=False):
    """losses: (K, 3) rows of (L+, L-, L0). Returns (status, c, w, curv)."""
    L = np.ascontiguousarray(losses, dtype=np.float64).reshape(-1, 3)
    K = L.shape[0]
    c = np.full(K, np.nan)
    w = np.full(K, np.nan)
    cv = np.full(K, np.nan)
    rc = lib().oracle_precondition(_ptr(L), K, eps, alpha, lambda_reg, int(one_sided), _ptr(c), _ptr(w), _ptr(cv))
    return rc, c, w, cv


def update(tensors, dtypes, seed, c, lr):
    n, ptrs, numel, dt = _table(tensors, dtypes)
    cc = np.ascontiguousarray(c, dtype=np.float64)
    rc = lib().oracle_update(n, ptrs, _ptr(numel), _ptr(dt), seed, _ptr(cc), len(cc), lr)
    if rc != OK:
        raise RuntimeError(f"oracle_update: {rc}")


def update_sequential(tensors, dtypes, seed, c, lr):
    n, ptrs, numel, dt = _table(tensors, dtypes)
    cc = np.ascontiguousarray(c, dtype=np.float64)
    rc = lib().oracle_update_sequential(n, ptrs, _ptr(numel), _ptr(dt), seed, _ptr(cc), len(cc), lr)
    if rc != OK:
        raise RuntimeError(f"oracle_update_sequential: {rc}")


def update_elements(dtype, g, theta, seed, c, lr):
    g = np.ascontiguousarray(g, dtype=np.uint64)
    th = np.ascontiguousarray(theta, dtype=np.float32)
    cc = np.ascontiguousarray(c, dtype=np.float64)
    out = np.zeros(len(g), dtype=np.uint32)
    rc = lib().oracle_update_elements(dtype, len(g), _ptr(g), _ptr(th), seed, _ptr(cc), len(cc), lr, _ptr(out))
    if rc != OK:
        raise RuntimeError(f"oracle_update_elements: {rc}")
    return out


def quadratic_loss(theta, a):
    th = np.ascontiguousarray(theta, dtype=np.float32)
    aa = np.ascontiguousarray(a, dtype=np.float32)
    assert th.size == aa.size
    return lib().oracle_quadratic_loss(_ptr(th), _ptr(aa), th.size)
