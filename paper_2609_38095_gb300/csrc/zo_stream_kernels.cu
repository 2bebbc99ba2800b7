// zo_stream_kernels.cu -- the HBM-streaming kernels of the 1.5-SPSA step:
// fused perturb (Algorithm 1, ApplyPackedPerturbation), the out-of-place pair
// of perturbations, fused K-probe update (Sec. 4.2, Eqs. 5-6) and the debug
// views of a probe.
//
// Work unit: one thread owns one 16-element Philox block at a time (grid-
// stride over the virtual block space of the launch's tensor table). A block
// of a 16-bit tensor is 32 bytes: one 256-bit load and one 256-bit store when
// the tensor is 32-byte aligned, element-wise access for a tensor's last,
// partial block. The perturbation passes and the update hand tensors that
// are not 32-byte aligned to perturb_shift_kernel / update_shift_kernel,
// which work on aligned 32-byte chunks straddling two blocks; the pair pass
// hands them (and fp32 tensors) to pair_shift_kernel when plus and minus
// share their offset, and takes narrower accesses otherwise.
#include "zo_device.cuh"

namespace zo {

// ---------------------------------------------------------------------------
// Perturb: theta <- rn(fp32(theta) + scale * z_k) in place.
//
// z_k[g] is bit `bit` of byte (g mod 16) of Philox(b = g/16, ctr2) (packing 1:
// ctr2 = k/8, bit = k mod 8; packing 8: ctr2 = k, bit = 0). Byte m sits at
// bits 8(m mod 4).. of word m/4; shifting the word left by
// 31 - 8(m mod 4) - bit puts the probe bit in the sign position, which then
// flips -scale into +scale (bit 1 -> z = +1). The product scale * z is exact,
// so the element result is one fp32 add and one rounding to storage.
//
// A launch may apply two perturbations in sequence (zo_perturb2): the value
// is rounded to storage after each, exactly as two separate passes would,
// but theta crosses HBM once.
// ---------------------------------------------------------------------------
// The same with the sign moved by a multiply (PerturbOp::mul), in the vector
// loops: it moves half of the sign injection from the integer ALU, the busiest
// pipe of these loops, to the multiply-add pipe (measured: single-op pass
// -1.1 to -1.7 % time on the OPT-30B / OPT-13B-shaped sets).
__device__ __forceinline__ uint32_t sign_bit_mul(const uint4& x, int i, const PerturbOp& op) {
  return (word_of(x, i >> 2) * op.mul[i & 3]) & 0x80000000u;
}

__device__ __forceinline__ float add_signed_mul(float th, const uint4& x, int i, const PerturbOp& op) {
  return __fadd_rn(th, __uint_as_float(op.nscale_bits ^ sign_bit_mul(x, i, op)));
}

// Sixteen 16-bit weights in registers (element 2r in the low half of v[r]).
// CROSS: a two-op pass whose probes fall in two groups of 8 (two Philox calls
// per block, one pass in eight of the fused schedule). Its adds are packed
// fp32x2 adds, the same round-to-nearest sum per element: with the second
// Philox call the loop is issue-bound and the packed adds take it from 20.5
// to 18.9 ms on the OPT-30B-shaped set, while the one-group pass, bound by
// HBM, is 1 % slower with them, so it keeps scalar adds.
template <uint8_t DT, int NOPS, bool CROSS = false>
__device__ __forceinline__ void perturb_regs16(uint32_t (&v)[8], const uint4 (&x)[2], const PerturbOp (&op)[2]) {
#pragma unroll
  for (int r = 0; r < 8; ++r) {
#pragma unroll
    for (int o = 0; o < NOPS; ++o) {
      if constexpr (CROSS) {
        float2 f = unpack2<DT>(v[r]);
        fadd2_rn(f.x, f.y, __uint_as_float(op[o].nscale_bits ^ sign_bit_mul(x[o], 2 * r, op[o])),
                 __uint_as_float(op[o].nscale_bits ^ sign_bit_mul(x[o], 2 * r + 1, op[o])));
        v[r] = pack2<DT>(f.x, f.y);
      } else {
        const float2 f = unpack2<DT>(v[r]);
        v[r] = pack2<DT>(add_signed_mul(f.x, x[o], 2 * r, op[o]), add_signed_mul(f.y, x[o], 2 * r + 1, op[o]));
      }
    }
  }
}

// A thread's position in the tensor table. Its blocks only move forward and
// usually stay inside one tensor, so the table is re-read only when a block
// leaves the current tensor.
struct Cursor {
  int t;           // tensor index
  uint32_t tb;     // first launch block of tensor t
  uint32_t te;     // one past its last block
  uint32_t n16;    // full blocks from tb on that take the pipelined 16-bit path (0 if it does not)
  uint32_t n32;    // the same for the pipelined fp32 path of the single-op loop
  uint16_t* tp;    // base pointer
  uint32_t vd;     // launch block minus virtual block (relative to blk_base) in tensor t
  uint8_t dt;      // storage dtype
};

// Launch blocks below tb (padding between tensors) give b - tb >= 2^31, so
// they fail both n16 and n32 tests and go to perturb_block_other, which skips
// them.
__device__ __forceinline__ void cursor_seek(const TensorTable& tab, Cursor& c, uint32_t b) {
  c.t = advance_tensor(tab, c.t, b);
  c.tb = tensor_blk_begin(tab, c.t);
  c.te = tab.blk_end[c.t];
  const uint8_t fl = tab.flags[c.t];
  c.dt = fl & kDtypeMask;
  // pipelined path: full, 32-byte aligned blocks of a 16-bit tensor
  const uint32_t full = static_cast<uint32_t>(tab.numel[c.t] / 16);
  c.n16 = ((fl & kVec32) && c.dt != kF32) ? full : 0u;
  c.n32 = ((fl & kVec32) && c.dt == kF32) ? full : 0u;
  c.tp = reinterpret_cast<uint16_t*>(tab.ptr[c.t]);
  c.vd = tab.vdelta[c.t];
}

// Any other block: fp32, a partial last block, or an unaligned tensor. One
// instantiation per calling kernel (TAG): ptxas 13.0 crashes when two kernels
// share this non-inlined function. Blocks of tensors flagged kShift are
// perturb_shift_kernel's and left alone (the loops above stay exactly as
// they are for the aligned tensors).
template <int NOPS, int TAG>
__device__ __noinline__ void perturb_block_other(const TensorTable& tab, int t, uint32_t b, uint4 x0, uint4 x1,
                                                 PerturbOp op0, PerturbOp op1) {
  const uint8_t fl = tab.flags[t];
  if ((fl & kShift) || b < tensor_blk_begin(tab, t)) return;  // perturb_shift_kernel's, or padding
  const int64_t e0 = static_cast<int64_t>(b - tensor_blk_begin(tab, t)) * 16;
  const int64_t cnt = min(static_cast<int64_t>(16), tab.numel[t] - e0);
  const uint8_t dt = fl & kDtypeMask;
  void* base = reinterpret_cast<void*>(tab.ptr[t]);
  if (cnt == 16 && (fl & kVec32) && dt == kF32) {
    float* p = static_cast<float*>(base) + e0;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      uint32_t v[8];
      ld256(p + 8 * half, v);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        float th = add_signed(__uint_as_float(v[r]), x0, 8 * half + r, op0);
        if (NOPS == 2) th = add_signed(th, x1, 8 * half + r, op1);
        v[r] = __float_as_uint(th);
      }
      st256(p + 8 * half, v);
    }
  } else if (cnt == 16 && dt != kF32) {  // a full block of an unaligned 16-bit tensor
    uint16_t* p = static_cast<uint16_t*>(base) + e0;
    uint32_t v[8];
    ld16x16(p, v);
    const uint4 x[2] = {x0, x1};
    const PerturbOp op[2] = {op0, op1};
    if (dt == kBF16)
      perturb_regs16<kBF16, NOPS>(v, x, op);
    else
      perturb_regs16<kF16, NOPS>(v, x, op);
    st16x16(p, v);
  } else {
    for (int i = 0; i < cnt; ++i) {
      float th = add_signed(load_elem(base, dt, e0 + i), x0, i, op0);
      if (NOPS == 2) th = add_signed(round_to_storage(dt, th), x1, i, op1);
      store_elem(base, dt, e0 + i, th);
    }
  }
}

// A run of n blocks of one 16-bit tensor, all full and 32-byte aligned, at
// p, p + pstride, ... with virtual blocks vb, vb + stride, ...: a tight,
// software-pipelined loop (the next block's 256-bit load is issued before the
// current block is computed and stored, so two loads per thread stay in
// flight; the pass is HBM-bound and needs the bytes in flight).
template <int NOPS, uint8_t DT, bool CROSS = false>
__device__ __forceinline__ void perturb_run16(uint16_t* p, uint32_t n, size_t pstride, int64_t vb,
                                              uint32_t stride, const PerturbOp (&op)[2], bool same_ctr,
                                              const RoundKeys& keys) {
  uint32_t v[8];
  ld256(p, v);
  for (uint32_t i = 0; i < n; ++i) {
    uint16_t* pn = p + pstride;
    uint32_t vn[8];
    if (i + 1 < n) ld256(pn, vn);
    uint4 x[2];
    x[0] = block_bits(vb, op[0].ctr2, keys);
    x[1] = x[0];
    if (NOPS == 2 && (CROSS || !same_ctr)) x[1] = block_bits(vb, op[1].ctr2, keys);
    perturb_regs16<DT, NOPS, CROSS>(v, x, op);
    st256(p, v);
    p = pn;
    vb += stride;
#pragma unroll
    for (int r = 0; r < 8; ++r) v[r] = vn[r];
  }
}

// Grid-stride over the launch's blocks, one block per iteration: the load of
// the thread's next block (through the cursor, in whatever tensor it lies) is
// issued before the current block is computed and stored. Every lane of a
// warp runs the same number of iterations, whatever the tensor sizes. With
// F32V (single-op launches that contain aligned fp32 tensors) full fp32
// blocks are pipelined too, as two 256-bit halves; otherwise they go to
// perturb_block_other, and the 16-bit path keeps its smaller register set.
enum : int { kBlockOther = 0, kBlock16 = 1, kBlock32 = 2 };

template <bool F32V>
__device__ __forceinline__ int block_kind(const Cursor& c, uint32_t b) {
  const uint32_t d = b - c.tb;
  if (d < c.n16) return kBlock16;
  if (F32V && d < c.n32) return kBlock32;
  return kBlockOther;
}

__device__ __forceinline__ void* block_addr(const Cursor& c, uint32_t b, int kind) {
  const size_t bytes = kind == kBlock32 ? 64 : 32;
  return reinterpret_cast<char*>(c.tp) + static_cast<size_t>(b - c.tb) * bytes;
}

template <int NOPS, bool F32V, bool CROSS = false>
__device__ __forceinline__ void perturb_blocks(const PerturbParams& P, const PerturbOp (&op)[2], bool same_ctr) {
  const TensorTable& tab = P.tab;
  const uint32_t blk_total = tab.blk_total;
  const uint32_t stride = gridDim.x * blockDim.x;
  uint32_t b = blockIdx.x * blockDim.x + threadIdx.x;  // launch-relative; < 2^31 + stride never wraps
  if (b >= blk_total) return;
  Cursor c;
  c.t = 0;
  cursor_seek(tab, c, b);
  int t = c.t;  // tensor and dtype of the current block
  uint8_t dt = c.dt;
  int kind = block_kind<F32V>(c, b);
  void* p = block_addr(c, b, kind);
  uint32_t vd = c.vd;
  uint32_t v[8], w[8];  // the block (16-bit), or its two halves (fp32)
  if (kind != kBlockOther) ld256(p, v);
  if (kind == kBlock32) ld256(static_cast<char*>(p) + 32, w);
  while (true) {
    const uint32_t bn = b + stride;
    int kindn = kBlockOther;
    void* pn = nullptr;
    uint32_t vn[8], wn[8];
    if (bn < blk_total) {
      if (bn >= c.te) cursor_seek(tab, c, bn);
      kindn = block_kind<F32V>(c, bn);
      pn = block_addr(c, bn, kindn);
      if (kindn != kBlockOther) ld256(pn, vn);
      if (kindn == kBlock32) ld256(static_cast<char*>(pn) + 32, wn);
    }
    const int64_t vb = tab.blk_base + (b - vd);  // virtual block: the Philox counter
    uint4 x[2];
    x[0] = block_bits(vb, op[0].ctr2, P.keys);
    x[1] = x[0];
    if (NOPS == 2 && (CROSS || !same_ctr)) x[1] = block_bits(vb, op[1].ctr2, P.keys);
    if (kind == kBlock16) {
      if (dt == kBF16)
        perturb_regs16<kBF16, NOPS, CROSS>(v, x, op);
      else
        perturb_regs16<kF16, NOPS, CROSS>(v, x, op);
      st256(p, v);
    } else if (F32V && kind == kBlock32) {
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        v[r] = __float_as_uint(add_signed_mul(__uint_as_float(v[r]), x[0], r, op[0]));
        w[r] = __float_as_uint(add_signed_mul(__uint_as_float(w[r]), x[0], 8 + r, op[0]));
      }
      st256(p, v);
      st256(static_cast<char*>(p) + 32, w);
    } else {
      // each kernel its own copy of the out-of-line routine
      perturb_block_other<NOPS, F32V ? 2 : (CROSS ? kLoopBlocks + 8 : kLoopBlocks)>(tab, t, b, x[0], x[1], op[0],
                                                                                   op[1]);
    }
    if (bn >= blk_total) break;
    b = bn;
    t = c.t;
    dt = c.dt;
    vd = c.vd;
    kind = kindn;
    p = pn;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      v[r] = vn[r];
      w[r] = wn[r];
    }
  }
}

// By runs: while a thread's next blocks (b, b + stride, ... below end) lie in
// the full, aligned 16-bit region of its current tensor they go through the
// tight loop of perturb_run16; any other block (fp32, a partial last block,
// an unaligned tensor) is handled on its own.
template <int NOPS, int TAG, bool CROSS = false>
__device__ __forceinline__ void perturb_runs_range(const PerturbParams& P, const PerturbOp (&op)[2], bool same_ctr,
                                                   uint32_t b, uint32_t end, uint32_t stride) {
  const TensorTable& tab = P.tab;
  Cursor c;
  c.t = 0;
  bool seeked = false;
  while (b < end) {
    if (!seeked || b >= c.te) {
      cursor_seek(tab, c, b);
      seeked = true;
    }
    const int64_t vb = tab.blk_base + (b - c.vd);  // virtual block: the Philox counter
    if (b - c.tb < c.n16) {
      const uint32_t stop = min(c.tb + c.n16, end);
      const uint32_t n = (stop - b + stride - 1) / stride;  // this thread's blocks in the region
      uint16_t* p = c.tp + static_cast<size_t>(b - c.tb) * 16;
      const size_t pstride = static_cast<size_t>(stride) * 16;
      if (c.dt == kBF16)
        perturb_run16<NOPS, kBF16, CROSS>(p, n, pstride, vb, stride, op, same_ctr, P.keys);
      else
        perturb_run16<NOPS, kF16, CROSS>(p, n, pstride, vb, stride, op, same_ctr, P.keys);
      b += n * stride;
    } else {
      uint4 x[2];
      x[0] = block_bits(vb, op[0].ctr2, P.keys);
      x[1] = x[0];
      if (NOPS == 2 && !same_ctr) x[1] = block_bits(vb, op[1].ctr2, P.keys);
      perturb_block_other<NOPS, TAG>(tab, c.t, b, x[0], x[1], op[0], op[1]);
      b += stride;
    }
  }
}

// Grid-stride by runs. Fewer instructions per block than perturb_blocks, but
// the lanes of a warp leave a run up to one iteration apart, which costs
// most where runs are short (tensors of a few blocks per thread).
template <int NOPS, bool CROSS = false>
__device__ __forceinline__ void perturb_runs(const PerturbParams& P, const PerturbOp (&op)[2], bool same_ctr) {
  const uint32_t stride = gridDim.x * blockDim.x;
  perturb_runs_range<NOPS, CROSS ? kLoopRuns + 8 : kLoopRuns, CROSS>(
      P, op, same_ctr, blockIdx.x * blockDim.x + threadIdx.x, P.tab.blk_total, stride);
}

// LOOP selects perturb_blocks (kLoopBlocks) or perturb_runs (kLoopRuns);
// CROSS marks a two-op launch whose probes fall in two groups of 8. The
// single-op pass (zo_perturb) always walks block by block (4.99 ms against
// 5.56 ms by runs on the Qwen3-8B-shaped set, equal elsewhere). For the two-op
// pass (zo_perturb2) the faster loop and grid depend on the parameter list
// (OPT-30B-shaped: runs with 3 blocks per SM 18.54 ms, per block with 4
// 18.72 ms; Qwen3-8B-shaped: 5.96 ms against 5.27 ms), so the host times the
// candidates on the caller's own list; all give the same bits.
template <int NOPS, int LOOP, bool F32V = false, bool CROSS = false>
__global__ void __launch_bounds__(256) perturb_kernel(const __grid_constant__ PerturbParams P) {
  if (P.status != nullptr && *P.status != 0) return;
  PerturbOp op[2] = {P.op[0], P.op[1]};
  if (P.coef != nullptr)
    op[0].nscale_bits = __float_as_uint(__double2float_rn(P.coef_mul * P.coef[P.probe])) ^ 0x80000000u;
  const bool same_ctr = op[1].ctr2 == op[0].ctr2;
  if (LOOP == kLoopBlocks)
    perturb_blocks<NOPS, F32V, CROSS>(P, op, same_ctr);
  else
    perturb_runs<NOPS, CROSS>(P, op, same_ctr);
}

// ---------------------------------------------------------------------------
// Unaligned tensors (kShift): the same perturbation over 32-byte aligned
// chunks instead of Philox blocks, so every full chunk moves with 256-bit
// accesses whatever the tensor's offset. Chunk c (elements 16c - a ..
// 16c - a + 15) draws its signs from bytes 16 - a .. 31 - a of the 32 bytes
// Philox(c - 1) ++ Philox(c). In a warp, lane l generates block
// c0 - 1 + l and works on chunk c0 - 1 + l with the block below taken from
// lane l - 1 by a shuffle: 32 Philox calls per 31 chunks, lane 0 only
// generates. Chunks that cross the tensor's ends go element by element.
// ---------------------------------------------------------------------------
// Bytes b .. b + 15 (b = 0..15) of the 32-byte string lo ++ hi.
__device__ __forceinline__ uint4 window16(const uint4& lo, const uint4& hi, uint32_t b) {
  const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
  uint32_t e[6], d[5];
#pragma unroll
  for (int i = 0; i < 6; ++i) e[i] = (b & 8u) ? w[i + 2] : w[i];  // move by two words
#pragma unroll
  for (int i = 0; i < 5; ++i) d[i] = (b & 4u) ? e[i + 1] : e[i];  // and by one
  const uint32_t sh = 8u * (b & 3u);
  return make_uint4(__funnelshift_r(d[0], d[1], sh), __funnelshift_r(d[1], d[2], sh),
                    __funnelshift_r(d[2], d[3], sh), __funnelshift_r(d[3], d[4], sh));
}

__device__ __forceinline__ uint4 shfl_up4(const uint4& x) {
  return make_uint4(__shfl_up_sync(0xffffffffu, x.x, 1), __shfl_up_sync(0xffffffffu, x.y, 1),
                    __shfl_up_sync(0xffffffffu, x.z, 1), __shfl_up_sync(0xffffffffu, x.w, 1));
}

// A chunk across an end of the tensor, element by element (not inlined: it
// is rare and would otherwise hold registers in the vector path).
template <int NOPS, uint8_t DT>
__device__ __noinline__ void shift_chunk_elements(void* base, int64_t n, int64_t e0, uint4 y0, uint4 y1,
                                                  PerturbOp op0, PerturbOp op1) {
  for (int p = 0; p < 16; ++p) {
    const int64_t e = e0 + p;
    if (e < 0 || e >= n) continue;
    float th = add_signed(load_elem(base, DT, e), y0, p, op0);
    if (NOPS == 2) th = add_signed(round_to_storage(DT, th), y1, p, op1);
    store_elem(base, DT, e, th);
  }
}

// Chunk c is the lane's own (lane > 0) and lies wholly inside the tensor.
__device__ __forceinline__ bool shift_full(int lane, int64_t c, uint32_t a, int64_t n) {
  return lane > 0 && c >= 1 && 16 * c - a + 16 <= n;
}

// One group of kShiftGroup chunks of tensor t (all lanes of the warp), as
// kShiftSub rounds of 31 chunks. 16-bit chunks are software-pipelined: the
// load of the lane's next chunk is issued before the current one is
// computed (two 32-byte loads in flight per lane, as for fp32's two halves).
template <int NOPS, uint8_t DT>
__device__ __forceinline__ void shift_group(const PerturbParams& P, const PerturbOp (&op)[2], bool same_ctr, int t,
                                            int64_t c_first) {
  constexpr int kElem = DT == kF32 ? 4 : 2;
  constexpr bool kAhead = DT != kF32;
  constexpr int kWords = 16 * kElem / 4;  // 32-bit words per chunk: 8 (16-bit) or 16 (fp32)
  const TensorTable& tab = P.tab;
  const uintptr_t ptr = tab.ptr[t];
  const int64_t n = tab.numel[t];
  const uint32_t a = static_cast<uint32_t>(ptr & 31u) / kElem;  // 1..15 (16-bit) or 1..7 (fp32)
  char* chunk0 = reinterpret_cast<char*>(ptr - (ptr & 31u));     // 32-byte aligned, a elements before the tensor
  const int64_t nchunks = (n + a + 15) / 16;
  const int64_t vb0 = virtual_block(tab, t, tensor_blk_begin(tab, t));  // virtual block of element 0
  const int lane = static_cast<int>(threadIdx.x & 31u);
  int64_t c = c_first + lane - 1;  // lane 0: the block below lane 1's chunk, no chunk of its own
  bool full = shift_full(lane, c, a, n);
  uint32_t v[kWords];
  if (kAhead && full) ld256(chunk0 + c * (16 * kElem), *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
#pragma unroll 1
  for (int s = 0; s < kShiftSub; ++s) {
    const int64_t cn = c + kShiftLanes;
    bool fulln = false;
    uint32_t vn[kWords];
    if (kAhead && s + 1 < kShiftSub) {
      fulln = shift_full(lane, cn, a, n);
      if (fulln) ld256(chunk0 + cn * (16 * kElem), *reinterpret_cast<uint32_t(*)[8]>(&vn[0]));
    }
    char* q = chunk0 + c * (16 * kElem);
    if (!kAhead && full) {
      ld256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
      ld256(q + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[kWords - 8]));
    }
    const int64_t vb = vb0 + c;
    uint4 x[2], y[2];
    x[0] = block_bits(vb, op[0].ctr2, P.keys);
    x[1] = x[0];
    if (NOPS == 2 && !same_ctr) x[1] = block_bits(vb, op[1].ctr2, P.keys);
    y[0] = window16(shfl_up4(x[0]), x[0], 16u - a);
    y[1] = y[0];
    if (NOPS == 2 && !same_ctr) y[1] = window16(shfl_up4(x[1]), x[1], 16u - a);
    if (full) {
      if constexpr (DT == kF32) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float th = add_signed_mul(__uint_as_float(v[i]), y[0], i, op[0]);
          if (NOPS == 2) th = add_signed_mul(th, y[1], i, op[1]);
          v[i] = __float_as_uint(th);
        }
        st256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
        st256(q + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[kWords - 8]));
      } else {
        perturb_regs16<DT, NOPS>(*reinterpret_cast<uint32_t(*)[8]>(&v[0]), y, op);
        st256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
      }
    } else if (lane > 0 && c >= 0 && c < nchunks) {
      shift_chunk_elements<NOPS, DT>(reinterpret_cast<void*>(ptr), n, 16 * c - a, y[0], y[1], op[0], op[1]);
    }
    c = cn;
    if (kAhead) {
      full = fulln;
#pragma unroll
      for (int r = 0; r < kWords; ++r) v[r] = vn[r];
    } else {
      full = shift_full(lane, c, a, n);
    }
  }
}

// One kernel per storage type (a shared one would hold the registers of all
// three paths): the host launches it for each type its unaligned tensors
// have, with grp_end counting only that type's tensors. Four blocks per SM
// (64 registers, no spills): measured faster than three (80 registers) for
// both the single- and the two-op pass.
template <int NOPS, uint8_t DT>
__global__ void __launch_bounds__(256, 4) perturb_shift_kernel(const __grid_constant__ ShiftParams S) {
  const PerturbParams& P = S.p;
  if (P.status != nullptr && *P.status != 0) return;
  PerturbOp op[2] = {P.op[0], P.op[1]};
  if (P.coef != nullptr)
    op[0].nscale_bits = __float_as_uint(__double2float_rn(P.coef_mul * P.coef[P.probe])) ^ 0x80000000u;
  const bool same_ctr = op[1].ctr2 == op[0].ctr2;
  const uint32_t warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
  int t = 0;
  for (uint32_t g = warp; g < S.grp_total; g += nwarps) {  // the same g on every lane of the warp
    while (g >= S.grp_end[t]) ++t;
    const int64_t c_first = static_cast<int64_t>(g - (t == 0 ? 0u : S.grp_end[t - 1])) * kShiftGroup;
    shift_group<NOPS, DT>(P, op, same_ctr, t, c_first);
  }
}

// ---------------------------------------------------------------------------
// Out-of-place pair: plus <- rn(fp32(theta) + v), minus <- rn(fp32(theta) - v)
// with v = scale z_k[g] (exact), theta untouched. One read of theta and two
// writes instead of the three read-modify-write passes of +eps / -2 eps /
// +eps, and both forward points are one rounding away from theta.
// ---------------------------------------------------------------------------
template <uint8_t DT>
__device__ __forceinline__ void pair_regs16(const uint32_t (&v)[8], const uint4& x, const PerturbOp& op,
                                            uint32_t (&p)[8], uint32_t (&m)[8]) {  // p may alias v
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const float2 f = unpack2<DT>(v[r]);
    const float d0 = __uint_as_float(op.nscale_bits ^ sign_bit_mul(x, 2 * r, op));
    const float d1 = __uint_as_float(op.nscale_bits ^ sign_bit_mul(x, 2 * r + 1, op));
    p[r] = pack2<DT>(__fadd_rn(f.x, d0), __fadd_rn(f.y, d1));
    m[r] = pack2<DT>(__fsub_rn(f.x, d0), __fsub_rn(f.y, d1));
  }
}

__device__ __noinline__ void pair_block_other(const PairTable& tab, int t, uint32_t b, uint4 x, PerturbOp op) {
  if (tab.flags[t] & kShift) return;  // pair_shift_kernel's
  const uint32_t tb = t == 0 ? 0u : tab.blk_end[t - 1];
  const int64_t e0 = static_cast<int64_t>(b - tb) * 16;
  const int cnt = b + 1 == tab.blk_end[t] ? tab.last[t] : 16;
  const uint8_t dt = tab.flags[t] & kDtypeMask;
  const void* src = reinterpret_cast<const void*>(tab.src[t]);
  void* pl = reinterpret_cast<void*>(tab.plus[t]);
  void* mi = reinterpret_cast<void*>(tab.minus[t]);
  if (cnt == 16 && dt != kF32) {  // a full block with an unaligned pointer among the three
    uint32_t v[8], m[8];
    ld16x16(static_cast<const uint16_t*>(src) + e0, v);
    if (dt == kBF16)
      pair_regs16<kBF16>(v, x, op, v, m);
    else
      pair_regs16<kF16>(v, x, op, v, m);
    st16x16(static_cast<uint16_t*>(pl) + e0, v);
    st16x16(static_cast<uint16_t*>(mi) + e0, m);
    return;
  }
  for (int i = 0; i < cnt; ++i) {
    const float th = load_elem(src, dt, e0 + i);
    const float d = __uint_as_float(op.nscale_bits ^ sign_bit(x, i, op.bit));
    store_elem(pl, dt, e0 + i, __fadd_rn(th, d));
    store_elem(mi, dt, e0 + i, __fsub_rn(th, d));
  }
}

// A thread's position in a pair table (as Cursor for TensorTable).
struct PairCursor {
  int t;
  uint32_t tb, te, tfe;  // first block, one past the last, one past the last full vector block (else tb)
  uint8_t dt;
};

__device__ __forceinline__ void pair_seek(const PairTable& tab, PairCursor& c, uint32_t b) {
  while (b >= tab.blk_end[c.t]) ++c.t;
  c.tb = c.t == 0 ? 0u : tab.blk_end[c.t - 1];
  c.te = tab.blk_end[c.t];
  c.dt = tab.flags[c.t] & kDtypeMask;
  c.tfe = ((tab.flags[c.t] & kVec32) && c.dt != kF32) ? c.te - (tab.last[c.t] < 16 ? 1u : 0u) : c.tb;
}

// Grid-stride one block per iteration, the next block's theta load issued
// before the current block is computed (the single-op perturb's loop).
__global__ void __launch_bounds__(256) perturb_pair_kernel(const __grid_constant__ PairParams P) {
  const PairTable& tab = P.tab;
  const PerturbOp op = P.op;
  const uint32_t stride = gridDim.x * blockDim.x;
  uint32_t b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= tab.blk_total) return;
  PairCursor c;
  c.t = 0;
  pair_seek(tab, c, b);
  int t = c.t;
  uint8_t dt = c.dt;
  size_t off = static_cast<size_t>(b - c.tb) * 16;
  bool vec = b < c.tfe;
  uint32_t v[8];
  if (vec) ld256(reinterpret_cast<const uint16_t*>(tab.src[t]) + off, v);
  while (true) {
    const uint32_t bn = b + stride;
    bool vecn = false;
    size_t offn = 0;
    uint32_t vn[8];
    if (bn < tab.blk_total) {
      if (bn >= c.te) pair_seek(tab, c, bn);
      vecn = bn < c.tfe;
      offn = static_cast<size_t>(bn - c.tb) * 16;
      if (vecn) ld256(reinterpret_cast<const uint16_t*>(tab.src[c.t]) + offn, vn);
    }
    const int64_t vb = tab.blk_base + b;
    const uint4 x = block_bits(vb, op.ctr2, P.keys);
    if (vec) {
      uint32_t m[8];
      if (dt == kBF16)
        pair_regs16<kBF16>(v, x, op, v, m);
      else
        pair_regs16<kF16>(v, x, op, v, m);
      st256(reinterpret_cast<uint16_t*>(tab.plus[t]) + off, v);
      st256(reinterpret_cast<uint16_t*>(tab.minus[t]) + off, m);
    } else {
      pair_block_other(tab, t, b, x, op);
    }
    if (bn >= tab.blk_total) break;
    b = bn;
    t = c.t;
    dt = c.dt;
    off = offn;
    vec = vecn;
#pragma unroll
    for (int r = 0; r < 8; ++r) v[r] = vn[r];
  }
}

// ---------------------------------------------------------------------------
// The pair of perturbations in 32-byte aligned chunks (as perturb_shift_kernel;
// a = 0 for aligned fp32 tensors, whose chunks are the blocks themselves).
// ---------------------------------------------------------------------------
template <uint8_t DT>
__device__ __noinline__ void pair_chunk_elements(const void* src, void* pl, void* mi, int64_t n, int64_t e0, uint4 y,
                                                 PerturbOp op) {
  for (int p = 0; p < 16; ++p) {
    const int64_t e = e0 + p;
    if (e < 0 || e >= n) continue;
    const float th = load_elem(src, DT, e);
    const float d = __uint_as_float(op.nscale_bits ^ sign_bit(y, p, op.bit));
    store_elem(pl, DT, e, __fadd_rn(th, d));
    store_elem(mi, DT, e, __fsub_rn(th, d));
  }
}

template <uint8_t DT>
__device__ __forceinline__ void pair_shift_group(const PairShiftParams& S, int t, int64_t c_first) {
  constexpr int kElem = DT == kF32 ? 4 : 2;
  constexpr bool kAhead = DT != kF32;
  constexpr int kWords = 16 * kElem / 4;
  const PerturbOp& op = S.op;
  const uintptr_t src = S.src[t];
  const uint32_t off = static_cast<uint32_t>(src & 31u);  // the same for plus and minus
  const uint32_t a = off / kElem;                        // 0..15 (16-bit) or 0..7 (fp32)
  const char* s0 = reinterpret_cast<const char*>(src - off);
  char* p0 = reinterpret_cast<char*>(S.plus[t] - off);
  char* m0 = reinterpret_cast<char*>(S.minus[t] - off);
  const int64_t n = S.numel[t];
  const int64_t nchunks = (n + a + 15) / 16;
  const int lane = static_cast<int>(threadIdx.x & 31u);
  auto full_at = [&](int64_t c) { return lane > 0 && 16 * c >= a && 16 * c - a + 16 <= n; };
  int64_t c = c_first + lane - 1;
  bool full = full_at(c);
  uint32_t v[kWords];
  if (kAhead && full) ld256(s0 + c * (16 * kElem), *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
#pragma unroll 1
  for (int s = 0; s < kShiftSub; ++s) {
    const int64_t cn = c + kShiftLanes;
    bool fulln = false;
    uint32_t vn[kWords];
    if (kAhead && s + 1 < kShiftSub) {
      fulln = full_at(cn);
      if (fulln) ld256(s0 + cn * (16 * kElem), *reinterpret_cast<uint32_t(*)[8]>(&vn[0]));
    }
    const int64_t cb = c * (16 * kElem);
    if (!kAhead && full) {
      ld256(s0 + cb, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
      ld256(s0 + cb + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[kWords - 8]));
    }
    const uint4 x = block_bits(S.vb0[t] + c, op.ctr2, S.keys);
    const uint4 below = shfl_up4(x);
    const uint4 y = a == 0 ? x : window16(below, x, 16u - a);
    if (full) {
      if constexpr (DT == kF32) {
        uint32_t m[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float th = __uint_as_float(v[i]);
          const float d = __uint_as_float(op.nscale_bits ^ sign_bit_mul(y, i, op));
          v[i] = __float_as_uint(__fadd_rn(th, d));
          m[i] = __float_as_uint(__fsub_rn(th, d));
        }
        st256(p0 + cb, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
        st256(p0 + cb + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[8]));
        st256(m0 + cb, *reinterpret_cast<uint32_t(*)[8]>(&m[0]));
        st256(m0 + cb + 32, *reinterpret_cast<uint32_t(*)[8]>(&m[8]));
      } else {
        uint32_t m[8];
        pair_regs16<DT>(*reinterpret_cast<uint32_t(*)[8]>(&v[0]), y, op, *reinterpret_cast<uint32_t(*)[8]>(&v[0]),
                        m);
        st256(p0 + cb, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
        st256(m0 + cb, m);
      }
    } else if (lane > 0 && c >= 0 && c < nchunks) {  // a chunk across an end of the tensor
      pair_chunk_elements<DT>(reinterpret_cast<const void*>(src), reinterpret_cast<void*>(S.plus[t]),
                              reinterpret_cast<void*>(S.minus[t]), n, 16 * c - a, y, op);
    }
    c = cn;
    if (kAhead) {
      full = fulln;
#pragma unroll
      for (int r = 0; r < kWords; ++r) v[r] = vn[r];
    } else {
      full = full_at(c);
    }
  }
}

// Bytes bo .. bo + 31 (bo even, 0..30) of the 64-byte string lo ++ hi.
__device__ __forceinline__ void window32(const uint32_t (&lo)[8], const uint32_t (&hi)[8], uint32_t bo,
                                         uint32_t (&out)[8]) {
  const uint32_t q = bo >> 2, sh = 8u * (bo & 3u);
  uint32_t e4[12], e2[10], e1[9];
#pragma unroll
  for (int i = 0; i < 12; ++i) {
    const uint32_t a = i < 8 ? lo[i] : hi[i - 8];
    const uint32_t b = i + 4 < 8 ? lo[i + 4] : hi[i - 4];
    e4[i] = (q & 4u) ? b : a;
  }
#pragma unroll
  for (int i = 0; i < 10; ++i) e2[i] = (q & 2u) ? e4[i + 2] : e4[i];
#pragma unroll
  for (int i = 0; i < 9; ++i) e1[i] = (q & 1u) ? e2[i + 1] : e2[i];
#pragma unroll
  for (int i = 0; i < 8; ++i) out[i] = __funnelshift_r(e1[i], e1[i + 1], sh);
}

// 16-bit tensors whose theta sits at another offset from the 32-byte grid
// than plus and minus: chunks follow the outputs, and theta's sixteen
// elements of chunk c are taken from the aligned 32-byte segments of theta
// that hold them (two, each also read by a neighbouring lane, whose second
// read hits L1; one when they fill a segment exactly).
template <uint8_t DT>
__device__ __forceinline__ void pair_shift_group_moved(const PairShiftParams& S, int t, int64_t c_first) {
  const PerturbOp& op = S.op;
  const uintptr_t src = S.src[t];
  const uint32_t off = static_cast<uint32_t>(S.plus[t] & 31u);  // the outputs' offset, shared by plus and minus
  const uint32_t a = off / 2, a_src = static_cast<uint32_t>(src & 31u) / 2;
  // theta element 16c - a sits at position d of theta's aligned segment c + dc
  const uint32_t d = (a_src + 16u - a) & 15u;
  const int64_t dc = a_src >= a ? 0 : -1;
  const char* s0 = reinterpret_cast<const char*>(src - (src & 31u));
  char* p0 = reinterpret_cast<char*>(S.plus[t] - off);
  char* m0 = reinterpret_cast<char*>(S.minus[t] - off);
  const int64_t n = S.numel[t];
  const int64_t nchunks = (n + a + 15) / 16;
  const int lane = static_cast<int>(threadIdx.x & 31u);
#pragma unroll 1
  for (int s = 0; s < kShiftSub; ++s) {
    const int64_t c = c_first + s * kShiftLanes + lane - 1;
    const bool full = lane > 0 && 16 * c >= a && 16 * c - a + 16 <= n;
    uint32_t lo[8], hi[8];
    if (full) {  // the second segment only when the sixteen elements reach into it (d > 0)
      const char* q = s0 + (c + dc) * 32;
      ld256(q, lo);
      if (d != 0) {
        ld256(q + 32, hi);
      } else {
#pragma unroll
        for (int r = 0; r < 8; ++r) hi[r] = lo[r];
      }
    }
    const uint4 x = block_bits(S.vb0[t] + c, op.ctr2, S.keys);
    const uint4 below = shfl_up4(x);
    const uint4 y = a == 0 ? x : window16(below, x, 16u - a);
    if (full) {
      uint32_t v[8], m[8];
      window32(lo, hi, 2u * d, v);
      pair_regs16<DT>(v, y, op, v, m);
      st256(p0 + c * 32, v);
      st256(m0 + c * 32, m);
    } else if (lane > 0 && c >= 0 && c < nchunks) {  // a chunk across an end of the tensor
      pair_chunk_elements<DT>(reinterpret_cast<const void*>(src), reinterpret_cast<void*>(S.plus[t]),
                              reinterpret_cast<void*>(S.minus[t]), n, 16 * c - a, y, op);
    }
  }
}

// MOVED: every tensor of the launch has theta at another offset than plus
// and minus (16-bit only); otherwise all three share it.
template <uint8_t DT, bool MOVED>
__global__ void __launch_bounds__(256, 4) pair_shift_kernel(const __grid_constant__ PairShiftParams S) {
  const uint32_t warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
  int t = 0;
  for (uint32_t g = warp; g < S.grp_total; g += nwarps) {  // the same g on every lane of the warp
    while (g >= S.grp_end[t]) ++t;
    const int64_t c_first = static_cast<int64_t>(g - (t == 0 ? 0u : S.grp_end[t - 1])) * kShiftGroup;
    if constexpr (MOVED)
      pair_shift_group_moved<DT>(S, t, c_first);
    else
      pair_shift_group<DT>(S, t, c_first);
  }
}

// ---------------------------------------------------------------------------
// Fused K-probe update: theta <- rn(fp32(theta) + sum_k a_k z_k[g]).
//
// Byte m of Philox(b, q) holds the signs of probes 8q..8q+7 for element
// 16b + m. Its low nibble indexes a 16-entry table of the fp32 partial sums
//   T[n] = ((s0 a_{4h} + s1 a_{4h+1}) + s2 a_{4h+2}) + s3 a_{4h+3},
//   s_j = +1 if bit j of n is set, else -1,
// for probe quad h = 2q, the high nibble the table of quad 2q + 1. Each
// element adds the two looked-up partials (low quad + high quad: the group's
// 8-probe partial) to its fp32 accumulator, groups in increasing order: one
// shared-memory load and one add per four probes instead of a select and an
// add per probe. Probes K..8*groups-1 have a = 0. update_lut8_kernel adds the
// same 8-probe partials in the same order, so both give the same bits.
//
// Shared-memory layout: probe group q owns a 256-byte frame starting on a
// 256-byte boundary of the shared window; bytes [0, 64) hold the table of
// quad 2q, [64, 128) the table of quad 2q + 1. Masking a Philox word once
// with 0x3C3C3C3C (after a shift by 2) leaves four nibble*4 offsets in its
// four bytes; one byte-permute then splices an offset under the frame's
// upper bytes, giving the lookup address in a single instruction.
// ---------------------------------------------------------------------------
constexpr uint32_t kFrameBytes = 256;

__device__ __forceinline__ float lds_lo(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}

__device__ __forceinline__ float lds_hi(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1+64];" : "=f"(v) : "r"(addr));
  return v;
}

__device__ __forceinline__ void accumulate_block(float (&acc)[16], int64_t b, const UpdateParams& P,
                                                 uint32_t lut_base) {
  const uint32_t blo = static_cast<uint32_t>(b), bhi = static_cast<uint32_t>(static_cast<uint64_t>(b) >> 32);
  uint32_t frame = lut_base;
  for (int q = 0; q < P.groups; ++q, frame += kFrameBytes) {
    const uint4 x = philox10(blo, bhi, static_cast<uint32_t>(q), 0u, P.keys);
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      const uint32_t w = word_of(x, m);
      const uint32_t lo4 = (w << 2) & 0x3C3C3C3Cu;  // byte j: 4 * low nibble of byte j of w
      const uint32_t hi4 = (w >> 2) & 0x3C3C3C3Cu;  // byte j: 4 * high nibble of byte j of w
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t sel = 0x7650u | static_cast<uint32_t>(j);  // byte j of the offsets, bytes 1-3 of the frame
        const float tlo = lds_lo(__byte_perm(lo4, frame, sel));
        const float thi = lds_hi(__byte_perm(hi4, frame, sel));
        acc[4 * m + j] = __fadd_rn(acc[4 * m + j], __fadd_rn(tlo, thi));
      }
    }
  }
}

// Packing 8: the sign of probe k is bit 0 of the element's byte of
// Philox(b, k). Eight outputs (probes 8f..8f+7) are folded into the same
// nibble layout as packing 1 -- bit 0 of every byte moved to bit i + 2 of the
// low (i < 4) or high (i >= 4) offset word -- and looked up in the same tables.
__device__ __forceinline__ void accumulate_block_p8(float (&acc)[16], int64_t b, const UpdateParams& P,
                                                    uint32_t lut_base) {
  const uint32_t blo = static_cast<uint32_t>(b), bhi = static_cast<uint32_t>(static_cast<uint64_t>(b) >> 32);
  uint32_t frame = lut_base;
  for (int f = 0; f < P.groups; ++f, frame += kFrameBytes) {
    uint32_t lo4[4] = {0u, 0u, 0u, 0u}, hi4[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint4 x = philox10(blo, bhi, static_cast<uint32_t>(8 * f + i), 0u, P.keys);
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const uint32_t bits = word_of(x, m) & 0x01010101u;
        if (i < 4)
          lo4[m] |= bits << (i + 2);
        else
          hi4[m] |= bits << (i - 2);
      }
    }
#pragma unroll
    for (int m = 0; m < 4; ++m) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t sel = 0x7650u | static_cast<uint32_t>(j);
        const float tlo = lds_lo(__byte_perm(lo4[m], frame, sel));
        const float thi = lds_hi(__byte_perm(hi4[m], frame, sel));
        acc[4 * m + j] = __fadd_rn(acc[4 * m + j], __fadd_rn(tlo, thi));
      }
    }
  }
}

template <int PACK>
__device__ __forceinline__ void accumulate_any(float (&acc)[16], int64_t b, const UpdateParams& P,
                                               uint32_t lut_base) {
  if constexpr (PACK == kPacking8)
    accumulate_block_p8(acc, b, P, lut_base);
  else
    accumulate_block(acc, b, P, lut_base);
}

// One full, 32-byte aligned block: theta (16-bit) is loaded before the probe
// loop so the load overlaps the arithmetic; the leading perturbation, when
// present, is applied and rounded to storage before the probe sum is added.
template <int PACK, uint8_t DT>
__device__ __forceinline__ void update_block_vec(void* base, int64_t e0, int64_t b, const UpdateParams& P,
                                                 uint32_t lut_base, bool do_sum) {
  float acc[16];
#pragma unroll
  for (int m = 0; m < 16; ++m) acc[m] = 0.0f;
  if constexpr (DT == kF32) {
    if (do_sum) accumulate_any<PACK>(acc, b, P, lut_base);
    uint4 xp = make_uint4(0u, 0u, 0u, 0u);
    if (P.has_pre) xp = block_bits(b, P.pre.ctr2, P.keys);
    float* p = static_cast<float*>(base) + e0;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      uint32_t v[8];
      ld256(p + 8 * half, v);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        float th = __uint_as_float(v[r]);
        if (P.has_pre) th = add_signed(th, xp, 8 * half + r, P.pre);
        if (do_sum) th = __fadd_rn(th, acc[8 * half + r]);
        v[r] = __float_as_uint(th);
      }
      st256(p + 8 * half, v);
    }
  } else {
    uint16_t* p = static_cast<uint16_t*>(base) + e0;
    uint32_t v[8];
    ld256(p, v);
    if (do_sum) accumulate_any<PACK>(acc, b, P, lut_base);
    uint4 xp = make_uint4(0u, 0u, 0u, 0u);
    if (P.has_pre) xp = block_bits(b, P.pre.ctr2, P.keys);
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      if (P.has_pre) v[r] = pre_regs16<DT>(v[r], xp, r, P.pre);
      if (do_sum) {
        const float2 f = unpack2<DT>(v[r]);
        v[r] = pack2<DT>(__fadd_rn(f.x, acc[2 * r]), __fadd_rn(f.y, acc[2 * r + 1]));
      }
    }
    st256(p, v);
  }
}

// Per-CTA prologue of the update kernels: a_k = fp32(coef_mul * c_k) for the
// K probes (zero-padded to 8 * groups) and the per-quad partial-sum tables in
// their frames. Returns false when the block has nothing to do (a failed
// preconditioner and no leading perturbation); do_sum is false when only the
// leading perturbation applies.
__device__ __forceinline__ bool update_prologue(const UpdateParams& P, unsigned char* smem, int& skip,
                                                uint32_t& lut_base, bool& do_sum) {
  float* a_s = reinterpret_cast<float*>(smem);  // 8 * groups coefficients (zero padded)
  const uint32_t smem_sh = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  lut_base = (smem_sh + 32u * P.groups + kFrameBytes - 1) & ~(kFrameBytes - 1);
  float* lut = reinterpret_cast<float*>(smem + (lut_base - smem_sh));  // generic view of the frames
  if (threadIdx.x == 0) skip = (P.status != nullptr && *P.status != 0);
  const int npad = 8 * P.groups;
  for (int k = threadIdx.x; k < npad; k += blockDim.x)
    a_s[k] = k < P.K ? __double2float_rn(P.coef_mul * P.coef[k]) : 0.0f;
  __syncthreads();
  if (skip && !P.has_pre) return false;
  do_sum = !skip;  // a failed preconditioner still gets the leading perturbation
  for (int e = threadIdx.x; e < 32 * P.groups; e += blockDim.x) {
    const int h = e >> 4, n = e & 15;
    const float* a = a_s + 4 * h;
    float s = (n & 1) ? a[0] : -a[0];
    s = __fadd_rn(s, (n & 2) ? a[1] : -a[1]);
    s = __fadd_rn(s, (n & 4) ? a[2] : -a[2]);
    s = __fadd_rn(s, (n & 8) ? a[3] : -a[3]);
    lut[(h >> 1) * (kFrameBytes / 4) + (h & 1) * 16 + n] = s;
  }
  __syncthreads();
  return true;
}

template <int PACK>
__global__ void __launch_bounds__(256) update_kernel(const __grid_constant__ UpdateParams P) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int skip;
  uint32_t lut_base;
  bool do_sum;
  if (!update_prologue(P, smem, skip, lut_base, do_sum)) return;

  const TensorTable& tab = P.tab;
  const uint32_t stride = gridDim.x * blockDim.x;
  int t = 0;
  for (uint32_t bl = blockIdx.x * blockDim.x + threadIdx.x; bl < tab.blk_total; bl += stride) {
    t = advance_tensor(tab, t, bl);
    const uint32_t tb = tensor_blk_begin(tab, t);
    if (bl < tb) continue;  // padding between tensors
    const int64_t e0 = static_cast<int64_t>(bl - tb) * 16;
    const int64_t b = virtual_block(tab, t, bl);  // the Philox counter
    const int64_t cnt = min(static_cast<int64_t>(16), tab.numel[t] - e0);
    const uint8_t fl = tab.flags[t];
    const uint8_t dt = fl & kDtypeMask;
    void* base = reinterpret_cast<void*>(tab.ptr[t]);
    if (cnt == 16 && (fl & kVec32)) {
      if (dt == kBF16)
        update_block_vec<PACK, kBF16>(base, e0, b, P, lut_base, do_sum);
      else if (dt == kF16)
        update_block_vec<PACK, kF16>(base, e0, b, P, lut_base, do_sum);
      else
        update_block_vec<PACK, kF32>(base, e0, b, P, lut_base, do_sum);
    } else if (!(fl & kShift)) {  // kShift: an unaligned tensor, update_shift_kernel's
      float acc[16];
#pragma unroll
      for (int m = 0; m < 16; ++m) acc[m] = 0.0f;
      if (do_sum) accumulate_any<PACK>(acc, b, P, lut_base);
      uint4 xp = make_uint4(0u, 0u, 0u, 0u);
      if (P.has_pre) xp = block_bits(b, P.pre.ctr2, P.keys);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (i < cnt) {
          float th = load_elem(base, dt, e0 + i);
          if (P.has_pre) th = round_to_storage(dt, add_signed(th, xp, i, P.pre));
          if (do_sum) th = __fadd_rn(th, acc[i]);
          store_elem(base, dt, e0 + i, th);
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Fused update of unaligned tensors (kShift), in the 32-byte aligned chunks of
// perturb_shift_kernel. Lane l sums the probes of block c = c0 - 1 + l (in
// block order, exactly as update_kernel does) and takes the sums of block
// c - 1 from lane l - 1; chunk c's sixteen sums are elements 16 - a .. 31 - a
// of the two blocks' sums, so every element gets the same fp32 value as in
// update_kernel.
// ---------------------------------------------------------------------------
// out[p] = (lo ++ hi)[s + p] for p = 0..15, s = 0..15: four stages of selects.
__device__ __forceinline__ void window16f(const float (&lo)[16], const float (&hi)[16], uint32_t s,
                                          float (&out)[16]) {
  float t8[24], t4[20], t2[18];
#pragma unroll
  for (int i = 0; i < 24; ++i) {
    const float a = i < 16 ? lo[i] : hi[i - 16];
    const float b = i + 8 < 16 ? lo[i + 8] : hi[i - 8];
    t8[i] = (s & 8u) ? b : a;
  }
#pragma unroll
  for (int i = 0; i < 20; ++i) t4[i] = (s & 4u) ? t8[i + 4] : t8[i];
#pragma unroll
  for (int i = 0; i < 18; ++i) t2[i] = (s & 2u) ? t4[i + 2] : t4[i];
#pragma unroll
  for (int i = 0; i < 16; ++i) out[i] = (s & 1u) ? t2[i + 1] : t2[i];
}

template <int PACK, uint8_t DT>
__device__ __forceinline__ void update_shift_group(const UpdateParams& P, uint32_t lut_base, bool do_sum, int t,
                                                   int64_t c_first) {
  constexpr int kElem = DT == kF32 ? 4 : 2;
  constexpr int kWords = 16 * kElem / 4;
  const TensorTable& tab = P.tab;
  const uintptr_t ptr = tab.ptr[t];
  const int64_t n = tab.numel[t];
  const uint32_t a = static_cast<uint32_t>(ptr & 31u) / kElem;
  char* chunk0 = reinterpret_cast<char*>(ptr - (ptr & 31u));
  const int64_t nchunks = (n + a + 15) / 16;
  const int64_t vb0 = virtual_block(tab, t, tensor_blk_begin(tab, t));
  const int lane = static_cast<int>(threadIdx.x & 31u);
#pragma unroll 1
  for (int s = 0; s < kShiftSub; ++s) {
    const int64_t c = c_first + s * kShiftLanes + lane - 1;
    const bool full = shift_full(lane, c, a, n);
    char* q = chunk0 + c * (16 * kElem);
    uint32_t v[kWords];
    if (full) {  // issued before the probe sums, which hide its latency
      ld256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
      if constexpr (DT == kF32) ld256(q + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[8]));
    }
    float own[16], below[16], sum[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) own[m] = 0.0f;
    if (do_sum) accumulate_any<PACK>(own, vb0 + c, P, lut_base);
#pragma unroll
    for (int m = 0; m < 16; ++m) below[m] = __shfl_up_sync(0xffffffffu, own[m], 1);
    window16f(below, own, 16u - a, sum);
    uint4 y = make_uint4(0u, 0u, 0u, 0u);
    if (P.has_pre) {
      const uint4 xp = block_bits(vb0 + c, P.pre.ctr2, P.keys);
      y = window16(shfl_up4(xp), xp, 16u - a);
    }
    if (full) {
      if constexpr (DT == kF32) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float th = __uint_as_float(v[i]);
          if (P.has_pre) th = add_signed(th, y, i, P.pre);
          if (do_sum) th = __fadd_rn(th, sum[i]);
          v[i] = __float_as_uint(th);
        }
        st256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
        st256(q + 32, *reinterpret_cast<uint32_t(*)[8]>(&v[8]));
      } else {
#pragma unroll
        for (int r = 0; r < 8; ++r) {
          if (P.has_pre) v[r] = pre_regs16<DT>(v[r], y, r, P.pre);
          if (do_sum) {
            const float2 f = unpack2<DT>(v[r]);
            v[r] = pack2<DT>(__fadd_rn(f.x, sum[2 * r]), __fadd_rn(f.y, sum[2 * r + 1]));
          }
        }
        st256(q, *reinterpret_cast<uint32_t(*)[8]>(&v[0]));
      }
    } else if (lane > 0 && c >= 0 && c < nchunks) {  // a chunk across an end of the tensor
      void* base = reinterpret_cast<void*>(ptr);
#pragma unroll
      for (int p = 0; p < 16; ++p) {
        const int64_t e = 16 * c - a + p;
        if (e < 0 || e >= n) continue;
        float th = load_elem(base, DT, e);
        if (P.has_pre) th = round_to_storage(DT, add_signed(th, y, p, P.pre));
        if (do_sum) th = __fadd_rn(th, sum[p]);
        store_elem(base, DT, e, th);
      }
    }
  }
}

template <int PACK, uint8_t DT>
__global__ void __launch_bounds__(256) update_shift_kernel(const __grid_constant__ UpdateShiftParams S) {
  const UpdateParams& P = S.u;
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int skip;
  uint32_t lut_base;
  bool do_sum;
  if (!update_prologue(P, smem, skip, lut_base, do_sum)) return;
  const uint32_t warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
  int t = 0;
  for (uint32_t g = warp; g < S.grp_total; g += nwarps) {  // the same g on every lane of the warp
    while (g >= S.grp_end[t]) ++t;
    const int64_t c_first = static_cast<int64_t>(g - (t == 0 ? 0u : S.grp_end[t - 1])) * kShiftGroup;
    update_shift_group<PACK, DT>(P, lut_base, do_sum, t, c_first);
  }
}

// ---------------------------------------------------------------------------
// Debug views: probe k packed one bit per element (Appendix F layout) and the
// unpacked int8 signs, over a range of the virtual index space.
// ---------------------------------------------------------------------------
__global__ void probe_bytes_kernel(RoundKeys keys, uint32_t q, uint32_t j, int64_t first, int64_t n, uint8_t* out) {
  const int64_t b_first = first >> 1, b_last = (first + n - 1) >> 1;  // packed bytes 2b, 2b+1 <- block b
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t b = b_first + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b <= b_last; b += stride) {
    const uint4 x = philox10(static_cast<uint32_t>(b), static_cast<uint32_t>(static_cast<uint64_t>(b) >> 32), q, 0u,
                             keys);
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int64_t jb = 2 * b + half;
      if (jb < first || jb >= first + n) continue;
      uint32_t v = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int m = 8 * half + i;
        v |= ((word_of(x, m >> 2) >> (8 * (m & 3) + j)) & 1u) << i;
      }
      out[jb - first] = static_cast<uint8_t>(v);
    }
  }
}

__global__ void probe_signs_kernel(RoundKeys keys, uint32_t q, uint32_t j, int64_t first, int64_t n, int8_t* out) {
  const int64_t b_first = first >> 4, b_last = (first + n - 1) >> 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t b = b_first + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b <= b_last; b += stride) {
    const uint4 x = philox10(static_cast<uint32_t>(b), static_cast<uint32_t>(static_cast<uint64_t>(b) >> 32), q, 0u,
                             keys);
#pragma unroll
    for (int m = 0; m < 16; ++m) {
      const int64_t g = 16 * b + m;
      if (g < first || g >= first + n) continue;
      const uint32_t bit = (word_of(x, m >> 2) >> (8 * (m & 3) + j)) & 1u;
      out[g - first] = bit ? static_cast<int8_t>(1) : static_cast<int8_t>(-1);
    }
  }
}

}  // namespace zo

// ---------------------------------------------------------------------------
// Launch wrappers.
// ---------------------------------------------------------------------------
#include "zo_launch.h"

namespace zo {

cudaError_t launch_perturb(const PerturbParams& p, int grid, int loop, bool f32v, cudaStream_t stream) {
  const bool cross = p.nops == 2 && p.op[0].ctr2 != p.op[1].ctr2;
  if (p.nops == 1 && f32v)
    perturb_kernel<1, kLoopBlocks, true><<<grid, kThreads, 0, stream>>>(p);
  else if (p.nops == 1)
    perturb_kernel<1, kLoopBlocks><<<grid, kThreads, 0, stream>>>(p);
  else if (loop == kLoopRuns && cross)
    perturb_kernel<2, kLoopRuns, false, true><<<grid, kThreads, 0, stream>>>(p);
  else if (loop == kLoopRuns)
    perturb_kernel<2, kLoopRuns><<<grid, kThreads, 0, stream>>>(p);
  else if (cross)
    perturb_kernel<2, kLoopBlocks, false, true><<<grid, kThreads, 0, stream>>>(p);
  else
    perturb_kernel<2, kLoopBlocks><<<grid, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

static_assert(sizeof(PairParams) <= 32764, "pair table exceeds the kernel parameter space");
static_assert(sizeof(ShiftParams) <= 32764 && sizeof(UpdateShiftParams) <= 32764 && sizeof(PairShiftParams) <= 32764,
              "shift table exceeds the kernel parameter space");
static_assert(sizeof(PerturbParams) <= 32764 && sizeof(UpdateParams) <= 32764,
              "tensor table exceeds the kernel parameter space");

template <int NOPS>
void launch_shift_nops(const ShiftParams& p, uint8_t dt, int grid, cudaStream_t stream) {
  if (dt == kBF16)
    perturb_shift_kernel<NOPS, kBF16><<<grid, kThreads, 0, stream>>>(p);
  else if (dt == kF16)
    perturb_shift_kernel<NOPS, kF16><<<grid, kThreads, 0, stream>>>(p);
  else
    perturb_shift_kernel<NOPS, kF32><<<grid, kThreads, 0, stream>>>(p);
}

cudaError_t launch_perturb_shift(const ShiftParams& p, uint8_t dt, int grid, cudaStream_t stream) {
  if (p.p.nops == 2)
    launch_shift_nops<2>(p, dt, grid, stream);
  else
    launch_shift_nops<1>(p, dt, grid, stream);
  return cudaGetLastError();
}

cudaError_t launch_pair_shift(const PairShiftParams& p, uint8_t dt, bool moved, int grid, cudaStream_t stream) {
  if (dt == kBF16 && moved)
    pair_shift_kernel<kBF16, true><<<grid, kThreads, 0, stream>>>(p);
  else if (dt == kF16 && moved)
    pair_shift_kernel<kF16, true><<<grid, kThreads, 0, stream>>>(p);
  else if (dt == kBF16)
    pair_shift_kernel<kBF16, false><<<grid, kThreads, 0, stream>>>(p);
  else if (dt == kF16)
    pair_shift_kernel<kF16, false><<<grid, kThreads, 0, stream>>>(p);
  else
    pair_shift_kernel<kF32, false><<<grid, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

template <int PACK>
void launch_update_shift_pack(const UpdateShiftParams& p, uint8_t dt, int grid, size_t smem, cudaStream_t stream) {
  if (dt == kBF16)
    update_shift_kernel<PACK, kBF16><<<grid, kThreads, smem, stream>>>(p);
  else if (dt == kF16)
    update_shift_kernel<PACK, kF16><<<grid, kThreads, smem, stream>>>(p);
  else
    update_shift_kernel<PACK, kF32><<<grid, kThreads, smem, stream>>>(p);
}

cudaError_t launch_update_shift(const UpdateShiftParams& p, uint8_t dt, int grid, cudaStream_t stream) {
  const size_t smem = update_smem_bytes(p.u.groups);
  if (p.u.packing == kPacking8)
    launch_update_shift_pack<kPacking8>(p, dt, grid, smem, stream);
  else
    launch_update_shift_pack<kPacking1>(p, dt, grid, smem, stream);
  return cudaGetLastError();
}

template <int PACK>
cudaError_t update_shift_bps_pack(int groups, uint8_t dt, int* out) {
  const size_t smem = update_smem_bytes(groups);
  if (dt == kBF16)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, update_shift_kernel<PACK, kBF16>, kThreads, smem);
  if (dt == kF16)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, update_shift_kernel<PACK, kF16>, kThreads, smem);
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, update_shift_kernel<PACK, kF32>, kThreads, smem);
}

cudaError_t update_shift_blocks_per_sm(int groups, int packing, uint8_t dt, int* out) {
  return packing == kPacking8 ? update_shift_bps_pack<kPacking8>(groups, dt, out)
                              : update_shift_bps_pack<kPacking1>(groups, dt, out);
}

cudaError_t launch_perturb_pair(const PairParams& p, int grid, cudaStream_t stream) {
  perturb_pair_kernel<<<grid, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

// Coefficients (32 bytes per group), alignment slack, one 256-byte frame per group.
size_t update_smem_bytes(int groups) { return static_cast<size_t>(groups) * (32 + kFrameBytes) + kFrameBytes; }

cudaError_t launch_update(const UpdateParams& p, int grid, cudaStream_t stream) {
  if (p.packing == kPacking8)
    update_kernel<kPacking8><<<grid, kThreads, update_smem_bytes(p.groups), stream>>>(p);
  else
    update_kernel<kPacking1><<<grid, kThreads, update_smem_bytes(p.groups), stream>>>(p);
  return cudaGetLastError();
}

cudaError_t perturb_blocks_per_sm(int nops, int loop, int* out) {
  if (nops == 1)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_kernel<1, kLoopBlocks>, kThreads, 0);
  if (loop == kLoopRuns)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_kernel<2, kLoopRuns>, kThreads, 0);
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_kernel<2, kLoopBlocks>, kThreads, 0);
}

template <int NOPS>
cudaError_t shift_bps_nops(uint8_t dt, int* out) {
  if (dt == kBF16)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_shift_kernel<NOPS, kBF16>, kThreads, 0);
  if (dt == kF16)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_shift_kernel<NOPS, kF16>, kThreads, 0);
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_shift_kernel<NOPS, kF32>, kThreads, 0);
}

cudaError_t shift_blocks_per_sm(int nops, uint8_t dt, int* out) {
  return nops == 2 ? shift_bps_nops<2>(dt, out) : shift_bps_nops<1>(dt, out);
}

cudaError_t pair_blocks_per_sm(int* out) {
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, perturb_pair_kernel, kThreads, 0);
}

cudaError_t update_blocks_per_sm(int groups, int packing, int* out) {
  if (packing == kPacking8)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, update_kernel<kPacking8>, kThreads,
                                                         update_smem_bytes(groups));
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, update_kernel<kPacking1>, kThreads,
                                                       update_smem_bytes(groups));
}

cudaError_t launch_probe_bytes(const RoundKeys& keys, uint32_t ctr2, uint32_t bit, int64_t first, int64_t n,
                               uint8_t* out, int grid, cudaStream_t stream) {
  probe_bytes_kernel<<<grid, kThreads, 0, stream>>>(keys, ctr2, bit, first, n, out);
  return cudaGetLastError();
}

cudaError_t launch_probe_signs(const RoundKeys& keys, uint32_t ctr2, uint32_t bit, int64_t first, int64_t n,
                               int8_t* out, int grid, cudaStream_t stream) {
  probe_signs_kernel<<<grid, kThreads, 0, stream>>>(keys, ctr2, bit, first, n, out);
  return cudaGetLastError();
}

}  // namespace zo
