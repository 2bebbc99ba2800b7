"""Python binding of libzo.so (include/zo.h): argument marshalling only.

Every numeric step runs in the library's CUDA kernels; this module turns torch
CUDA tensors into pointers, passes the current torch stream, and raises on a
non-zero status. There is no CPU path: if libzo.so is missing, every call
raises.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libzo.so")

ZO_OK = 0
ZO_ERR_ARG = -1
ZO_ERR_DTYPE = -2
ZO_ERR_ALIGN = -3
ZO_ERR_NONFINITE = -4
ZO_ERR_CUDA = -5
ZO_ERR_TOO_MANY_PROBES = -6
ZO_ERR_WORKSPACE = -7
ZO_MAX_PROBES = 1024
ZO_PRECOND_ONE_SIDED = 1
ZO_PRECOND_RELATIVE_CURVATURE = 2

DTYPE_CODE = {torch.float32: 0, torch.bfloat16: 1, torch.float16: 2}

EXPORTS = ["zo_status_string", "zo_last_cuda_error", "zo_version", "zo_set_packing", "zo_get_packing",
           "zo_perturb", "zo_perturb2", "zo_perturb_pair", "zo_precondition",
           "zo_precondition_ex", "zo_update", "zo_update_ex", "zo_update_sequential", "zo_probe_bytes", "zo_probe_signs",
           "zo_quadratic_loss_workspace_size", "zo_quadratic_loss", "zo_quadratic_loss_static",
           "zo_perturb_quadratic_loss_workspace_size", "zo_perturb_quadratic_loss"]
ZO_QUADRATIC_LOSS_STATIC_MAX_N = 8388608


class zo_tensor(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("numel", ctypes.c_int64), ("dtype", ctypes.c_int32),
                ("packing", ctypes.c_int32)]


class ZoError(RuntimeError):
    def __init__(self, fn, status):
        msg = f"{fn}: {status_string(status)}"
        if status == ZO_ERR_CUDA:
            msg += f" [{_lib().zo_last_cuda_error().decode()}]"
        super().__init__(msg)
        self.status = status


_L = None


def _lib():
    global _L
    if _L is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run paper_2609_38095_gb300.build.build() "
                               "(there is no fallback implementation)")
        L = ctypes.CDLL(LIB_PATH)
        c = ctypes
        vp, i32, i64, u32, u64, f32, f64 = c.c_void_p, c.c_int32, c.c_int64, c.c_uint32, c.c_uint64, c.c_float, c.c_double
        sig = {
            "zo_status_string": ([c.c_int], c.c_char_p),
            "zo_last_cuda_error": ([], c.c_char_p),
            "zo_version": ([], c.c_int),
            "zo_set_packing": ([i32], c.c_int),
            "zo_get_packing": ([], c.c_int),
            "zo_perturb": ([vp, i32, u64, u32, f32, vp], c.c_int),
            "zo_perturb2": ([vp, i32, u64, u32, f32, u32, f32, vp], c.c_int),
            "zo_perturb_pair": ([vp, vp, vp, i32, u64, u32, f32, vp], c.c_int),
            "zo_update_ex": ([vp, i32, u64, vp, i32, f64, vp, i32, u32, f32, vp], c.c_int),
            "zo_precondition": ([vp, i32, f64, vp, vp, vp], c.c_int),
            "zo_precondition_ex": ([vp, i32, f64, f64, f64, i32, vp, vp, vp, vp, vp], c.c_int),
            "zo_update": ([vp, i32, u64, vp, i32, f64, vp, vp], c.c_int),
            "zo_update_sequential": ([vp, i32, u64, vp, i32, f64, vp, vp], c.c_int),
            "zo_probe_bytes": ([u64, u32, i64, i64, vp, vp], c.c_int),
            "zo_probe_signs": ([u64, u32, i64, i64, vp, vp], c.c_int),
            "zo_quadratic_loss_workspace_size": ([i64], i64),
            "zo_quadratic_loss": ([vp, vp, i64, vp, vp, i64, vp], c.c_int),
            "zo_quadratic_loss_static": ([vp, vp, i64, vp, vp], c.c_int),
            "zo_perturb_quadratic_loss_workspace_size": ([i64], i64),
            "zo_perturb_quadratic_loss": ([vp, vp, i64, u64, i32, i32, u32, f32, u32, f32, vp, i32, i64, vp, i64, vp],
                                          c.c_int),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _L = L
    return _L


def status_string(status: int) -> str:
    return _lib().zo_status_string(int(status)).decode()


def version() -> int:
    return _lib().zo_version()


def set_packing(bits_per_value: int):
    """Probe packing of every later call: 1 (default) or 8 generated bits per
    weight and probe (zo_set_packing)."""
    _check("zo_set_packing", _lib().zo_set_packing(int(bits_per_value)))


def get_packing() -> int:
    return _lib().zo_get_packing()


class packing:
    """Context manager: run a block of calls under one probe packing."""

    def __init__(self, bits_per_value):
        self.bits = bits_per_value

    def __enter__(self):
        self.prev = get_packing()
        set_packing(self.bits)
        return self

    def __exit__(self, *exc):
        set_packing(self.prev)
        return False


def _check(fn, rc):
    if rc != ZO_OK:
        raise ZoError(fn, rc)


# The current stream's handle without building a torch Stream object (about
# 3 us of a 9 us call otherwise); the public route where torch lacks it.
_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _index(device):
    return device.index if device.index is not None else torch.cuda.current_device()


def _stream(device):
    idx = _index(device)
    if _raw_stream is not None:
        return ctypes.c_void_p(_raw_stream(idx))
    return ctypes.c_void_p(torch.cuda.current_stream(idx).cuda_stream)


class _on:
    """Makes `device` current for a call (the library launches on the current
    device); a no-op when it already is, the usual case."""
    __slots__ = ("idx", "prev")

    def __init__(self, device):
        self.idx = _index(device)
        self.prev = None

    def __enter__(self):
        cur = torch.cuda.current_device()
        if cur != self.idx:
            self.prev = cur
            torch.cuda.set_device(self.idx)
        return self

    def __exit__(self, *exc):
        if self.prev is not None:
            torch.cuda.set_device(self.prev)
        return False


def _dev_ptr(t, dtype=None, what="tensor"):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{what} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{what} must be {dtype}, got {t.dtype}")
    return ctypes.c_void_p(t.data_ptr())


def _same_device(dev, **tensors):
    """Raise unless every tensor lives on `dev` (the launch runs there)."""
    for name, t in tensors.items():
        if isinstance(t, torch.Tensor) and t.device != dev:
            raise ValueError(f"{name} is on {t.device}, the weights on {dev}")


class ParamList:
    """The parameter list of a training step: a fixed, ordered list of CUDA
    tensors, each updated in place. Build it once and pass it to every call of
    every step: the probes are defined by each element's position in it.
    packing (1 or 8) fixes the list's probe packing; None follows the process
    default (set_packing) at each call."""

    def __init__(self, tensors, packing=None):
        if packing not in (None, 1, 8):
            raise ValueError("packing must be None, 1 or 8")
        self.packing = packing
        self.tensors = list(tensors)
        n = len(self.tensors)
        arr = (zo_tensor * max(n, 1))()
        dev = None
        for i, t in enumerate(self.tensors):
            if not isinstance(t, torch.Tensor) or not t.is_cuda:
                raise TypeError("parameters must be CUDA tensors")
            if not t.is_contiguous():
                raise ValueError("parameters must be contiguous")
            if t.dtype not in DTYPE_CODE:
                raise TypeError(f"unsupported parameter dtype {t.dtype}")
            if dev is None:
                dev = t.device
            elif t.device != dev:
                raise ValueError("all parameters must live on one device")
            arr[i].ptr = t.data_ptr()
            arr[i].numel = t.numel()
            arr[i].dtype = DTYPE_CODE[t.dtype]
            arr[i].packing = packing or 0
        self._arr = arr
        self.n = n
        self.device = dev if dev is not None else torch.device("cuda", torch.cuda.current_device())

    @property
    def numels(self):
        return [t.numel() for t in self.tensors]

    def __len__(self):
        return self.n


def _plist(params):
    return params if isinstance(params, ParamList) else ParamList(params)


def perturb(params, seed: int, probe: int, scale: float):
    """theta <- theta + scale * z_probe in place (zo_perturb)."""
    p = _plist(params)
    with _on(p.device):
        _check("zo_perturb", _lib().zo_perturb(p._arr, p.n, seed, probe, scale, _stream(p.device)))


def perturb2(params, seed: int, probe_a: int, scale_a: float, probe_b: int, scale_b: float):
    """perturb(probe_a, scale_a) then perturb(probe_b, scale_b), bit for bit, in
    one pass over theta (zo_perturb2)."""
    p = _plist(params)
    with _on(p.device):
        _check("zo_perturb2", _lib().zo_perturb2(p._arr, p.n, seed, probe_a, scale_a, probe_b, scale_b,
                                                 _stream(p.device)))


def perturb_pair(params, plus, minus, seed: int, probe: int, scale: float):
    """plus <- theta + scale z_k and minus <- theta - scale z_k, both rounded
    once to storage, theta untouched, in one pass (zo_perturb_pair). plus and
    minus are lists of tensors shaped like params (same numel and dtype)."""
    p, pl, mi = _plist(params), _plist(plus), _plist(minus)
    if not (pl.n == mi.n == p.n):
        raise ValueError("plus and minus must have one tensor per parameter")
    if (pl.n and pl.device != p.device) or (mi.n and mi.device != p.device):
        raise ValueError("plus and minus must live on the parameters' device")
    with _on(p.device):
        _check("zo_perturb_pair", _lib().zo_perturb_pair(p._arr, pl._arr, mi._arr, p.n, seed, probe, scale,
                                                         _stream(p.device)))


def precondition(losses, eps: float, alpha: float = 0.1, lambda_reg: float = 1.0, one_sided: bool = False,
                 out=None, with_weights: bool = False, relative: bool = False, flags=None):
    """losses: CUDA float64 tensor (K, 3) of rows (L+, L-, L0).
    one_sided / relative set ZO_PRECOND_ONE_SIDED / ZO_PRECOND_RELATIVE_CURVATURE
    (`flags`, the raw bit word, overrides both when given).
    Returns (c, status) -- or (c, status, w, curv) with with_weights -- as CUDA
    tensors; status[0] is ZO_OK or ZO_ERR_NONFINITE once the kernel has run."""
    if flags is None:
        flags = (ZO_PRECOND_ONE_SIDED if one_sided else 0) | (ZO_PRECOND_RELATIVE_CURVATURE if relative else 0)
    if losses.dim() != 2 or losses.shape[1] != 3:
        raise ValueError("losses must have shape (K, 3)")
    lp = _dev_ptr(losses, torch.float64, "losses")
    K = losses.shape[0]
    dev = losses.device
    if out is None:
        c = torch.empty(K, dtype=torch.float64, device=dev)
        status = torch.empty(1, dtype=torch.int32, device=dev)
    else:
        c, status = out
        if c.numel() < K or status.numel() < 1:
            raise ValueError("out must be (c with at least K elements, status with at least one)")
    w = curv = None
    if with_weights:
        w = torch.empty(K, dtype=torch.float64, device=dev)
        curv = torch.empty(K, dtype=torch.float64, device=dev)
    with _on(dev):
        rc = _lib().zo_precondition_ex(lp, K, eps, alpha, lambda_reg, int(flags),
                                       _dev_ptr(c, torch.float64, "c"),
                                       _dev_ptr(w, torch.float64) if w is not None else None,
                                       _dev_ptr(curv, torch.float64) if curv is not None else None,
                                       _dev_ptr(status, torch.int32, "status"), _stream(dev))
    _check("zo_precondition", rc)
    return (c, status, w, curv) if with_weights else (c, status)


def update(params, seed: int, c, lr: float, status=None, pre=None):
    """theta <- theta - (lr / K) * sum_k c_k z_k in one pass (zo_update).
    pre=(probe, scale) first applies perturb(probe, scale) in the same pass
    (zo_update_ex), e.g. the last probe's restore."""
    p = _plist(params)
    st = _dev_ptr(status, torch.int32, "status") if status is not None else None
    has_pre, pre_probe, pre_scale = (0, 0, 0.0) if pre is None else (1, int(pre[0]), float(pre[1]))
    with _on(p.device):
        rc = _lib().zo_update_ex(p._arr, p.n, seed, _dev_ptr(c, torch.float64, "c"), c.numel(), lr, st,
                                 has_pre, pre_probe, pre_scale, _stream(p.device))
    _check("zo_update", rc)


def update_sequential(params, seed: int, c, lr: float, status=None):
    """Algorithm 1's K-pass application, the comparator (zo_update_sequential)."""
    p = _plist(params)
    st = _dev_ptr(status, torch.int32, "status") if status is not None else None
    with _on(p.device):
        rc = _lib().zo_update_sequential(p._arr, p.n, seed, _dev_ptr(c, torch.float64, "c"), c.numel(), lr, st,
                                         _stream(p.device))
    _check("zo_update_sequential", rc)


def probe_bytes(seed: int, probe: int, first: int, n: int, device=None):
    """Probe `probe` packed one bit per element (bytes first..first+n-1)."""
    out = torch.empty(n, dtype=torch.uint8, device=device or "cuda")
    with _on(out.device):
        rc = _lib().zo_probe_bytes(seed, probe, first, n, ctypes.c_void_p(out.data_ptr()), _stream(out.device))
    _check("zo_probe_bytes", rc)
    return out


def probe_signs(seed: int, probe: int, first: int, n: int, device=None):
    """z_probe[g] as int8 for g = first..first+n-1."""
    out = torch.empty(n, dtype=torch.int8, device=device or "cuda")
    with _on(out.device):
        rc = _lib().zo_probe_signs(seed, probe, first, n, ctypes.c_void_p(out.data_ptr()), _stream(out.device))
    _check("zo_probe_signs", rc)
    return out


def quadratic_loss_workspace_size(n: int) -> int:
    return _lib().zo_quadratic_loss_workspace_size(n)


def quadratic_loss(theta, a, out=None, workspace=None):
    """f = 1/2 sum a_i theta_i^2 in fp64, into out (a CUDA float64 tensor of
    one element, returned)."""
    n = theta.numel()
    if a.numel() != n:
        raise ValueError("theta and a differ in size")
    dev = theta.device
    if out is None:
        out = torch.empty(1, dtype=torch.float64, device=dev)
    if workspace is None:
        workspace = torch.empty(quadratic_loss_workspace_size(n), dtype=torch.uint8, device=dev)
    if out.numel() < 1:
        raise ValueError("out must hold one float64")
    _same_device(dev, a=a, out=out, workspace=workspace)
    with _on(dev):
        rc = _lib().zo_quadratic_loss(_dev_ptr(theta, torch.float32, "theta"), _dev_ptr(a, torch.float32, "a"), n,
                                      _dev_ptr(out, torch.float64, "out"), _dev_ptr(workspace, what="workspace"),
                                      workspace.numel() * workspace.element_size(), _stream(dev))
    _check("zo_quadratic_loss", rc)
    return out


class QuadraticLoss:
    """quadratic_loss with theta, a and the workspace checked once: a call
    takes only the address of its output (a float64 on theta's device, for
    example an element of a loss table) and enqueues the kernels. For a step
    that evaluates the loss 2K + 1 times on the same weights."""

    def __init__(self, theta, a, workspace=None):
        n = theta.numel()
        if a.numel() != n:
            raise ValueError("theta and a differ in size")
        self.device = theta.device
        if workspace is None:
            workspace = torch.empty(quadratic_loss_workspace_size(n), dtype=torch.uint8, device=self.device)
        if workspace.numel() * workspace.element_size() < quadratic_loss_workspace_size(n):
            raise ValueError("workspace too small")
        _same_device(self.device, a=a, workspace=workspace)
        self._keep = (theta, a, workspace)   # the addresses below stay valid while these live
        self._args = (_dev_ptr(theta, torch.float32, "theta"), _dev_ptr(a, torch.float32, "a"), n)
        self._ws = (_dev_ptr(workspace, what="workspace"), workspace.numel() * workspace.element_size())

    def out_address(self, out):
        """The address to pass for `out` (a float64 element on theta's device)."""
        if not isinstance(out, torch.Tensor) or out.dtype != torch.float64 or out.numel() < 1:
            raise ValueError("out must hold one float64")
        _same_device(self.device, out=out)
        return out.data_ptr()

    def __call__(self, out_address: int):
        with _on(self.device):
            rc = _lib().zo_quadratic_loss(*self._args, ctypes.c_void_p(out_address), *self._ws, _stream(self.device))
        _check("zo_quadratic_loss", rc)


def quadratic_loss_static(theta, a, out=None):
    """zo_quadratic_loss_static: the same loss with the library's fixed
    scratch instead of a workspace (the call itself allocates nothing; pass
    `out` to avoid the one allocation this wrapper would make)."""
    n = theta.numel()
    if a.numel() != n:
        raise ValueError("theta and a differ in size")
    dev = theta.device
    if out is None:
        out = torch.empty(1, dtype=torch.float64, device=dev)
    if out.numel() < 1:
        raise ValueError("out must hold one float64")
    _same_device(dev, a=a, out=out)
    with _on(dev):
        rc = _lib().zo_quadratic_loss_static(_dev_ptr(theta, torch.float32, "theta"), _dev_ptr(a, torch.float32, "a"),
                                             n, _dev_ptr(out, torch.float64, "out"), _stream(dev))
    _check("zo_quadratic_loss_static", rc)
    return out


def perturb_quadratic_loss_workspace_size(n: int) -> int:
    return _lib().zo_perturb_quadratic_loss_workspace_size(n)


def _quad_ops(ops):
    ops = list(ops)
    if len(ops) > 2:
        raise ValueError("at most two perturbations per pass")
    pa, sa = ops[0] if ops else (0, 0.0)
    pb, sb = ops[1] if len(ops) == 2 else (0, 0.0)
    return len(ops), int(pa), float(sa), int(pb), float(sb)


class QuadraticPass:
    """zo_perturb_quadratic_loss with theta, a and the workspace checked once:
    one forward point of the small workload per call -- up to two
    perturbations of theta (as perturb / perturb2 apply them) and the loss of
    the result, in one pass. The workspace is allocated zero-filled here, as
    the call requires. packing: None follows the process default."""

    def __init__(self, theta, a, workspace=None, packing=None):
        n = theta.numel()
        if a.numel() != n:
            raise ValueError("theta and a differ in size")
        if packing not in (None, 1, 8):
            raise ValueError("packing must be None, 1 or 8")
        self.device = theta.device
        size = perturb_quadratic_loss_workspace_size(n)
        if workspace is None:
            workspace = torch.zeros(size, dtype=torch.uint8, device=self.device)
        if workspace.numel() * workspace.element_size() < size:
            raise ValueError("workspace too small")
        _same_device(self.device, a=a, workspace=workspace)
        self._keep = (theta, a, workspace)
        self._args = (_dev_ptr(theta, torch.float32, "theta"), _dev_ptr(a, torch.float32, "a"), n)
        self._ws = (_dev_ptr(workspace, what="workspace"), workspace.numel() * workspace.element_size())
        self.packing = packing or 0

    def out_address(self, out):
        """The address to pass for `out` (float64 elements on theta's device)."""
        if not isinstance(out, torch.Tensor) or out.dtype != torch.float64 or out.numel() < 1:
            raise ValueError("out must hold float64 elements")
        _same_device(self.device, out=out)
        return out.data_ptr()

    def __call__(self, seed: int, ops, out_address: int, copies: int = 1, stride: int = 1):
        """ops: a list of at most two (probe, scale) pairs applied in order;
        the loss goes to copies float64 cells stride elements apart."""
        nops, pa, sa, pb, sb = _quad_ops(ops)
        with _on(self.device):
            rc = _lib().zo_perturb_quadratic_loss(*self._args, seed, self.packing, nops, pa, sa, pb, sb,
                                                  ctypes.c_void_p(out_address), copies, stride, *self._ws,
                                                  _stream(self.device))
        _check("zo_perturb_quadratic_loss", rc)


def perturb_quadratic_loss(theta, a, seed: int, ops, out=None, workspace=None, packing=None):
    """One pass: theta <- theta + scale z_probe for each (probe, scale) of ops
    (at most two, in order), then out[0] <- 1/2 sum a_i theta_i^2 of the
    result (zo_perturb_quadratic_loss). Returns out (a float64 tensor)."""
    if out is None:
        out = torch.empty(1, dtype=torch.float64, device=theta.device)
    q = QuadraticPass(theta, a, workspace=workspace, packing=packing)
    q(seed, ops, q.out_address(out))
    return out
