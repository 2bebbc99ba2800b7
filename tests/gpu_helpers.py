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
    with np.errstate(over="ignore", invalid="ignore"):   # infinities have no spacing
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
        with np.errstate(over="ignore", invalid="ignore"):
            return np.spacing(x.astype(np.float16)).astype(np.float64)
    # bf16: 8 significand bits, fp32's exponent range
    e = np.floor(np.log2(np.maximum(x, 2.0 ** -126)))
    return 2.0 ** (e - 7)


def update_error(dt, c, lr, want):
    """Largest |acc32 - A| + half an fp32 ulp of the result that the kernel's
    arithmetic allows, per element: A = sum_k a_k z_k (the oracle forms it
    exactly), acc32 the kernel's fp32 sum: per probe group of eight, two
    4-probe partials (three fp32 adds each) and their sum, added to the
    accumulator in group order (ceil(K/8) additions), so the recursive
    summation bound gives |acc32 - A| <= (ceil(K/8) + 3) u S <= (H + 2) u S
    with H = 2 ceil(K/8), S = sum |a_k| and u = 2^-24 (the larger H + 2 is
    used); fp32(theta + acc32) adds half an fp32 ulp."""
    K = len(c)
    H = 2 * ((K + 7) // 8)
    S = float(np.abs(update_coeffs(c, lr).astype(np.float64)).sum())
    return (H + 2) * 2.0 ** -24 * S + 0.5 * ulp_f32(want)


def update_bound(got, want, dt, c, lr):
    """Largest |gpu - oracle| the arithmetic allows for the fused update.

    Oracle: one rounding of theta + A (A exact). Kernel: fp32(theta + acc32),
    then, for 16-bit storage, one rounding to storage. Hence
      |gpu - oracle| <= ulp_s(gpu)/2 + ulp_s(oracle)/2 + update_error
    (fp32 storage: the storage rounding is the fp32 one already counted)."""
    e = update_error(dt, c, lr, want)
    if dt == W.DT_F32:
        return 1.0001 * (0.5 * ulp_f32(want) + e)
    return 1.0001 * (0.5 * (ulp_storage(got, dt) + ulp_storage(want, dt)) + e)


def assert_update_close(got_bits, want_bits, dt, c, lr, context=""):
    """Fused-update parity against the oracle, element by element.

    NaN where the oracle has NaN, with the same bits. bf16 / fp16 storage:
    every element within one ulp of the oracle, except in the cancellation
    band -- elements where half a storage ulp of the oracle's value is below
    the fp32 summation error (|theta + A| of the order of 2^p times that
    error), where no fp32 accumulation can promise one storage ulp -- which
    must meet the derived bound instead. fp32 storage: the derived bound.
    Returns counts (elements, bit-equal, largest ulp distance, band elements)."""
    gb = np.asarray(got_bits, dtype=np.uint32)
    wb = np.asarray(want_bits, dtype=np.uint32)
    g = bits_to_f64(gb, dt)
    w = bits_to_f64(wb, dt)
    nan_w, nan_g = np.isnan(w), np.isnan(g)
    bad = np.nonzero(nan_w != nan_g)[0]
    assert bad.size == 0, (context, "NaN mismatch", [(int(i), hex(int(gb[i])), hex(int(wb[i]))) for i in bad[:5]])
    bad = np.nonzero(nan_w & (gb != wb))[0]
    assert bad.size == 0, (context, "NaN encoding", [(int(i), hex(int(gb[i])), hex(int(wb[i]))) for i in bad[:5]])
    fin = ~nan_w
    g, w, gb, wb = g[fin], w[fin], gb[fin], wb[fin]
    bound = update_bound(g, w, dt, c, lr)
    if dt == W.DT_F32:
        band = np.ones(g.size, dtype=bool)
        ulp = np.zeros(g.size, dtype=np.int64)
    else:
        band = 0.5 * ulp_storage(w, dt) < update_error(dt, c, lr, w)
        ulp = ulp_distance16(gb, wb)
        far = np.nonzero(~band & (ulp > 1))[0]
        assert far.size == 0, (context, "more than one ulp outside the cancellation band",
                               [(int(i), hex(int(gb[i])), hex(int(wb[i])), int(ulp[i])) for i in far[:5]])
    # in the band (every element for fp32 storage) the derived bound; equal
    # infinities pass (their difference is NaN)
    with np.errstate(invalid="ignore"):
        bad = np.nonzero(band & ~((np.abs(g - w) <= bound) | (gb == wb)))[0]
    assert bad.size == 0, (context, [(int(i), g[i], w[i], bound[i]) for i in bad[:5]])
    return {"n": int(gb.size + np.sum(nan_w)), "equal": int(np.sum(gb == wb) + np.sum(nan_w)),
            "max_ulp": int(ulp.max()) if ulp.size else 0, "band": int(np.sum(band)) if dt != W.DT_F32 else 0}


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
