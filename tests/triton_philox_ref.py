"""Independent Philox4x32-10 outputs from Triton's ``tl.philox``, evaluated by
Triton's CPU interpreter (no GPU needed). Used only to pin the oracle.

Run as a script with TRITON_INTERPRET=1:
    python triton_philox_ref.py in.npz out.npy
in.npz holds ``seeds`` (uint64, S) and ``ctr`` (uint32, S x N x 4); out.npy
receives the S x N x 4 uint32 outputs.
"""
import os
import sys

import numpy as np


def main(src, dst):
    assert os.environ.get("TRITON_INTERPRET") == "1"
    import torch
    import triton
    import triton.language as tl

    @triton.jit
    def philox_kernel(seed, c0p, c1p, c2p, c3p, o0p, o1p, o2p, o3p, N: tl.constexpr):
        i = tl.arange(0, N)
        c0 = tl.load(c0p + i)
        c1 = tl.load(c1p + i)
        c2 = tl.load(c2p + i)
        c3 = tl.load(c3p + i)
        r0, r1, r2, r3 = tl.philox(seed, c0, c1, c2, c3)
        tl.store(o0p + i, r0)
        tl.store(o1p + i, r1)
        tl.store(o2p + i, r2)
        tl.store(o3p + i, r3)

    data = np.load(src)
    seeds = data["seeds"].astype(np.uint64)
    ctr = data["ctr"].astype(np.uint32)
    S, N, _ = ctr.shape
    assert N & (N - 1) == 0, "N must be a power of two"
    out = np.zeros_like(ctr)
    for s in range(S):
        cs = [torch.from_numpy(np.ascontiguousarray(ctr[s, :, j]).view(np.int32)) for j in range(4)]
        os_ = [torch.zeros(N, dtype=torch.int32) for _ in range(4)]
        philox_kernel[(1,)](int(seeds[s]), *cs, *os_, N=N)
        for j in range(4):
            out[s, :, j] = os_[j].numpy().view(np.uint32)
    np.save(dst, out)


if __name__ == "__main__":
    main(sys.argv[1], sys.argv[2])
