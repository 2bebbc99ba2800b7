"""Helpers shared by the GPU parity tests: storage round-trips between torch
tensors and the oracle's numpy storage arrays, ulp distances and bounds."""
import numpy as np
import torch

from paper_2609_38095_gb300 import workloads as W

TORCH_TO_DT = {torch.float32: W.DT_F32, torch.bfloat16: W.DT_BF16, torch.float16: W.DT_F16}


def storage_np(t: torch.Tensor) -> np.ndarray:
    """Raw storage of a tensor as numpy: float32, or uint16 bit patterns."""
    c = t.detach().cpu()
    if c.dtype == torch.float32:
        return c.numpy().copy()
    return c.view(torch.int16).numpy().view(np.uint16).copy()


def storage_bits(t) -> np.ndarray:
    """Bit patterns as uint32 (fp32 bits, or 16-bit patterns zero-extended)."""
    a = storage_np(t) if isinstance(t, torch.Tensor) else t
    return a.view(np.uint32).copy() if a.dtype == np.float32 else a.astype(np.uint32)


def to_torch(a: np.ndarray, dtype, device="cuda") -> torch.Tensor:
    if dtype == torch.float32:
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(dtype).to(device)


def bits_to_f64(bits: np.ndarray, dt: int) -> np.ndarray:
    bits = np.asarray(bits, dtype=np.uint32)
    if dt == W.DT_F32:
        return bits.view(np.float32).astype(np.float64)
    if dt == W.DT_BF16:
        return (bits << 16).view(np.float32).astype(np.float64)
    return bits.astype(np.uint16).view(np.float16).astype(np.float64)


def ulp_distance16(a_bits, b_bits) -> np.ndarray:
    """Distance in units in the last place between two 16-bit patterns of the
    same format (sign-magnitude order; +0 and -0 coincide)."""
    def key(b):
        b = np.asarray(b, dtype=np.int64)
        mag = b & 0x7FFF
        return np.where(b & 0x8000, -mag, mag)
    return np.abs(key(a_bits) - key(b_bits))


def ulp_f32(x) -> np.ndarray:
    return np.spacing(np.abs(np.asarray(x, dtype=np.float32))).astype(np.float64)


def update_coeffs(c, lr):
    m = -(lr / len(c))
    return np.array([np.float32(m * ci) for ci in c], dtype=np.float32)


def ulp_storage(x, dt) -> np.ndarray:
    """Spacing of the storage format at |x| (subnormal spacing near zero)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    if dt == W.DT_F32:
        return ulp_f32(x)
    if dt == W.DT_F16:
        return np.spacing(x.astype(np.float16)).astype(np.float64)
    # bf16: 8 significand bits, fp32's exponent range
    e = np.floor(np.log2(np.maximum(x, 2.0 ** -126)))
    return 2.0 ** (e - 7)


def update_bound(got, want, dt, c, lr):
    """Largest |gpu - oracle| the arithmetic allows for the fused update.

    Oracle: one rounding of theta + A (A = sum_k a_k z_k, exact).
    Kernel: acc = A + e with |e| <= (H + 2) u S (4-probe partials of 3 fp32
    adds, H = 2 ceil(K/8) partials added in order, S = sum |a_k|, u = 2^-24);
    then fp32(theta + acc) (half an fp32 ulp) and, for 16-bit storage, one
    more rounding (half a storage ulp). Hence
      |gpu - oracle| <= ulp_s(gpu)/2 + ulp_s(oracle)/2 + ulp32(gpu)/2 + (H+3) u S
    which is one storage ulp unless theta + A nearly cancels."""
    K = len(c)
    H = 2 * ((K + 7) // 8)
    S = float(np.abs(update_coeffs(c, lr).astype(np.float64)).sum())
    b = 0.5 * (ulp_storage(got, dt) + ulp_storage(want, dt)) + (H + 3) * 2.0 ** -24 * S
    if dt != W.DT_F32:
        b = b + 0.5 * ulp_f32(got)
    return 1.0001 * b


def assert_update_close(got_bits, want_bits, dt, c, lr, context="", min_one_ulp=0.999):
    """Every element within the derived bound; for bf16 / fp16 storage also at
    least `min_one_ulp` of the elements within one ulp of the storage format
    (fp32 storage has no one-ulp bar: its fp32 accumulation error is of the
    order of an fp32 ulp of sum |a_k|)."""
    g = bits_to_f64(got_bits, dt)
    w = bits_to_f64(want_bits, dt)
    bound = update_bound(g, w, dt, c, lr)
    bad = np.nonzero(~(np.abs(g - w) <= bound))[0]
    assert bad.size == 0, (context, [(int(i), g[i], w[i], bound[i]) for i in bad[:5]])
    if dt != W.DT_F32 and g.size >= 1000:   # the one-ulp bar is stated for bf16 / fp16 storage
        one = ulp_distance16(got_bits, want_bits) <= 1
        assert np.mean(one) >= min_one_ulp, (context, float(np.mean(one)))


def sample_positions(numels, n_random=1 << 16, seed=0):
    """(tensor index, element index) pairs: ends of every tensor + uniform."""
    numels = np.asarray(numels, dtype=np.int64)
    cum = np.concatenate([[0], np.cumsum(numels)])
    rng = np.random.default_rng(seed)
    flat = rng.integers(0, cum[-1], n_random)
    t_r = np.searchsorted(cum, flat, side="right") - 1
    i_r = flat - cum[t_r]
    ts, is_ = [t_r], [i_r]
    for t, n in enumerate(numels):
        if n == 0:
            continue
        e = np.unique(np.concatenate([np.arange(min(16, n)), np.arange(max(0, n - 16), n)]))
        ts.append(np.full(e.size, t))
        is_.append(e)
    t_all = np.concatenate(ts)
    i_all = np.concatenate(is_)
    order = np.lexsort((i_all, t_all))
    return t_all[order], i_all[order]


def gather(params, t_idx, i_idx):
    """Storage bits and fp32 values of the sampled elements."""
    out_bits, out_f32 = [], []
    bounds = np.flatnonzero(np.diff(np.concatenate([[-1], t_idx, [len(params)]])))
    for a, b in zip(bounds[:-1], bounds[1:]):
        t = int(t_idx[a])
        idx = torch.from_numpy(i_idx[a:b]).to(params[t].device)
        v = params[t][idx]
        out_f32.append(v.float().cpu().numpy())
        out_bits.append(storage_bits(v))
    return np.concatenate(out_bits), np.concatenate(out_f32)
